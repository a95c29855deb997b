// frt_attention.cu — chunk flash attention over the rolling KV cache on sm_103a.
//
// out[i,h,:] = sum_j softmax_j(scale * <q_i, k_j>) v_j over every valid cache row j
// (the whole window is visible to every query of the chunk: bidirectional within the
// chunk, all earlier chunks of the window), bf16 operands, fp32 accumulation.
//
// One CTA = one work item = (stream, head, 256 query rows as two 128-row tiles, a range of
// the KV tiles: all of them, or one of n_split parts for the groups of the last waves).
// Three warpgroups (384 threads, one CTA per SM); registers are rebalanced with
// setmaxnreg: warpgroup 0 drops to kRegsCtl, the two softmax warpgroups rise to kRegsSm.
//   warp 0      TMA producer: Q tiles once, then K/V tiles (K0, V0, K1, V1, ...) through
//               a STAGES-deep shared-memory ring.
//   warp 1      TMEM allocator + tcgen05.mma issuer (converged warp, lane 0 issues):
//                 S_g  = Q_g K_j^T  A, B from shared memory (K-major, 128-byte swizzle)
//                 O_g += P_g V_j    A = P from TMEM, B = V from shared memory (MN-major)
//               issued as PV_0(j), S_0(j+1), PV_1(j), S_1(j+1): the tiles alternate
//   warp 2      observer: waits on the K/V barriers the issuer needs next and hands
//               off to it through a named barrier; the softmax groups meet the issuer at
//               their own named barriers when P is in TMEM (the issuer touches no mbarrier
//               in the KV loop)
//   warp 3      idle
//   warps 4-7   softmax group 0 (query tile 0), one thread per query row
//   warps 8-11  softmax group 1 (query tile 1)
// TMEM (512 columns): S_0 [0,128), S_1 [128,256), O_0 [256,256+D), O_1 [256+D,256+2D).
// P_g (bf16 pairs) overwrites the first 64 columns of S_g once the scores are in
// registers. PV_g(j) is issued before S_g(j+1); tcgen05.mma from one thread executes
// in issue order, so S_g(j+1) never overwrites P_g(j) early, and the arrival of S_g(j)
// implies PV_g(j-1) is complete (so O_g may be rescaled then). While one tile's softmax
// runs, the tensor pipe works on the other tile's PV and next S.
// The softmax exponentiates against a stale reference max in the log2 domain and
// rescales O only when a row's sum signals possible overflow (O and the row sum share
// the reference, so the result is exact).
//
// Every wait is bounded (mbar_wait): a role that gives up records FRT_ERR_TIMEOUT in the
// stream's status block, raises a CTA-wide abort flag, and the CTA drains its in-flight
// TMA/MMA work (bounded) and frees TMEM before exiting.
#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {

namespace {

constexpr int kThreads = 384;
// Register split: 128 threads x kRegsCtl + 256 threads x kRegsSm must equal the launch
// allocation 384 x kRegsLaunch (checked on the host before every first launch).
constexpr int kRegsLaunch = 168;
constexpr int kRegsCtl = 104;
constexpr int kRegsSm = 200;
static_assert(128 * kRegsCtl + 256 * kRegsSm == kThreads * kRegsLaunch, "register split");
constexpr int kBM = 128;   // query rows per tile
constexpr int kBN = 128;   // KV rows per tile
constexpr float kOverflowGuard = 1.152921504606846976e18f;   // 2^60
constexpr int kTimeoutCode = 6;  // FRT_ERR_TIMEOUT
// Named barriers: 0 __syncthreads, 1-3 the softmax groups' epilogues, 4 the issuer /
// observer hand-off (warps 1 and 2), 5 and 6 P_0 and P_1 ready (softmax group g's 128
// threads and the issuer warp's 32).
constexpr int kBarHandoff = 4;
constexpr int kBarP = 5;

template <int D>
struct Cfg {
    static constexpr int NCB = D / 64;                 // 128-byte column blocks per row
    static constexpr int Q_TILE = kBM * D * 2;
    static constexpr int KV_TILE = kBN * D * 2;
    static constexpr int STAGES = (D == 128) ? 5 : 8;
    static constexpr int OFF_Q = 0;
    static constexpr int OFF_KV = OFF_Q + 2 * Q_TILE;
    static constexpr int OFF_BAR = OFF_KV + STAGES * KV_TILE;
    static constexpr int SMEM = OFF_BAR + 256 + 1024;  // barriers + alignment slack
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(kBM, kBN, false);
    static constexpr uint32_t IDESC_O = idesc_bf16_f32(kBM, D, true);
};

struct Bars {
    uint64_t q_full;
    uint64_t q_ready[2];
    uint64_t s_full[2];
    uint64_t o_done[2];
    uint64_t drain[2];
    uint64_t kv_full[8];
    uint64_t step_done[4];
    uint64_t k0_done;
    uint64_t epi_full[2];
    uint32_t tmem_base;
    int abort_flag;
    int last_split;
};

__device__ __forceinline__ void report(DeviceStatus* st, volatile int* abort, int role, int where) {
    *abort = 1;
    if (st != nullptr) {
        volatile DeviceStatus* s = st;
        if (s->code == 0) {
            s->block = blockIdx.x;
            s->role = role;
            s->where = where;
            __threadfence_system();
            s->code = kTimeoutCode;
        }
    }
}

template <int D, int MAXS, bool ROPE>
__global__ void __launch_bounds__(kThreads, 1)
attn_kernel(const __grid_constant__ AttnParams<MAXS> p) {
    using C = Cfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    Bars* bars = reinterpret_cast<Bars*>(smem + C::OFF_BAR);
    const uint32_t sQ = smem_u32(smem + C::OFF_Q);
    const uint32_t sKV = smem_u32(smem + C::OFF_KV);
    volatile int* abort = &bars->abort_flag;

    // ---- work item ---------------------------------------------------------------------
    // Query groups (stream, head, 256 query rows) are numbered in launch order: streams in
    // the host's order, then head-major. Groups [0, n_full) are one item each; every later
    // group (the tail) is cut into n_split items over contiguous KV-tile ranges, whose
    // unnormalised partials the last of them to finish merges. Cutting only the tail fills
    // the last wave without paying the partials' round trip on every group.
    const int item = blockIdx.x;
    int group, split, n_parts;
    if (item < p.n_full) {
        group = item;
        split = 0;
        n_parts = 1;
    } else {
        const int v = item - p.n_full;
        const int tg = v / p.n_split;
        group = p.n_full + tg;
        split = v - tg * p.n_split;
        n_parts = p.n_split;
    }
    const int tail = group - p.n_full;                         // tail group index (n_parts > 1)
    int si = 0;
    while (si + 1 < p.n_streams && group >= p.s[si + 1].group_begin) ++si;
    const AttnStreamDesc& sd = p.s[si];
    const int local = group - sd.group_begin;
    const int head = local / sd.n_qpairs;
    const int pair = local - head * sd.n_qpairs;
    const int m0 = pair * (2 * kBM);
    const bool active1 = (m0 + kBM) < sd.n_q;
    const int ng = active1 ? 2 : 1;
    const int tiles_total = (sd.n_kv + kBN - 1) / kBN;
    const int t0 = split * tiles_total / n_parts;            // this item's KV tiles
    const int n_tiles = (split + 1) * tiles_total / n_parts - t0;
    const int n_loads = 2 * n_tiles;
#ifdef FRT_DEBUG
    // every index this item derives must lie inside the launch's extents; an item that
    // fails records FRT_ERR_BOUNDS and exits before it touches memory (the whole CTA
    // returns here, before any barrier or TMEM allocation)
    if (item >= p.total_items || group < 0 || group >= p.groups_total || si >= p.n_streams ||
        head < 0 || head >= p.heads || pair < 0 || pair >= sd.n_qpairs || n_tiles < 1 ||
        t0 < 0 || t0 + n_tiles > tiles_total ||
        (n_parts > 1 && (tail < 0 || tail >= p.tails_cap ||
                         (long long)(tail + 1) * n_parts * 2 * kBM > p.part_rows_cap))) {
        if (threadIdx.x == 0) record_status(p.status, kStatusBounds, 9, item);
        return;
    }
#endif

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bars->q_full), 1);
        for (int g = 0; g < 2; ++g) {
            mbar_init(smem_u32(&bars->q_ready[g]), kBM);
            mbar_init(smem_u32(&bars->s_full[g]), 1);
            mbar_init(smem_u32(&bars->o_done[g]), 1);
        }
        mbar_init(smem_u32(&bars->drain[0]), 1);
        mbar_init(smem_u32(&bars->drain[1]), 1);
        for (int s = 0; s < C::STAGES; ++s) mbar_init(smem_u32(&bars->kv_full[s]), 1);
        for (int s = 0; s < 4; ++s) mbar_init(smem_u32(&bars->step_done[s]), 1);
        mbar_init(smem_u32(&bars->k0_done), 1);
        mbar_init(smem_u32(&bars->epi_full[0]), 1);
        mbar_init(smem_u32(&bars->epi_full[1]), 1);
        bars->abort_flag = 0;
        fence_mbar_init();
        fence_proxy_async_smem();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&bars->tmem_base), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    const uint64_t lim = p.wait_limit_ns;

    if (warp < 4) {
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsCtl));
      if (warp == 0) {
        // ================================ TMA producer =================================
        if (lane == 0) {
            tma_prefetch_map(&sd.q_map);
            tma_prefetch_map(&sd.k_map);
            tma_prefetch_map(&sd.v_map);
            const uint32_t qbar = smem_u32(&bars->q_full);
            mbar_arrive_expect_tx(qbar, ng * C::Q_TILE);
            for (int g = 0; g < ng; ++g)
                for (int cb = 0; cb < C::NCB; ++cb)
                    tma_load_3d(sQ + g * C::Q_TILE + cb * (kBM * 128), &sd.q_map, qbar,
                                cb * 64, head, m0 + g * kBM);
            // Load L reuses the ring slot of load L - STAGES. Slots are released per KV
            // step: step j reads V_j and K_{j+1} (loads 2j+1, 2j+2) and its single release
            // commit arrives on step_done[j % 4]; K_0 (load 0) is released by k0_done.
            // The MMA thread issues that commit early in step j+1 (inside PV_0(j+1), which
            // needs only loads up to 2j+4, whose slots step j-1 released). Step j+4's
            // commit needs loads the producer has not issued while it waits for step j,
            // so the parity of step_done[j % 4] is never ambiguous.
            int L = 0;
            for (; L < n_loads; ++L) {
                const int stage = L % C::STAGES;
                if (L >= C::STAGES) {
                    const int prev = L - C::STAGES;
                    bool got;
                    if (prev == 0) {
                        got = mbar_wait(smem_u32(&bars->k0_done), 0, lim, abort);
                    } else {
                        const int step = (prev - 1) >> 1;
                        got = mbar_wait(smem_u32(&bars->step_done[step & 3]), (step >> 2) & 1,
                                        lim, abort);
                    }
                    if (!got) {
                        report(p.status, abort, 0, L);
                        break;
                    }
                }
                const CUtensorMap* map = (L & 1) ? &sd.v_map : &sd.k_map;
                const int row = (t0 + (L >> 1)) * kBN;
                // K_j and V_j (loads 2j, 2j+1) complete on one barrier, kv_full[j % 4]:
                // the MMA thread then tests one barrier per KV step instead of two
                const uint32_t fb = smem_u32(&bars->kv_full[(L >> 1) & 3]);
                if ((L & 1) == 0) mbar_arrive_expect_tx(fb, 2 * C::KV_TILE);
                const uint32_t dst = sKV + stage * C::KV_TILE;
                for (int cb = 0; cb < C::NCB; ++cb)
                    tma_load_3d(dst + cb * (kBN * 128), map, fb, cb * 64, head, row);
            }
            // drain: every issued load must have landed before the CTA may exit (a pair
            // left half-issued by an error completes only by the wait's time limit)
            const int npairs = (L + 1) >> 1;
            for (int pr = (npairs > 4 ? npairs - 4 : 0); pr < npairs; ++pr)
                mbar_wait_drain(smem_u32(&bars->kv_full[pr & 3]), (pr >> 2) & 1, lim);
            mbar_wait_drain(qbar, 0, lim);
        }
      } else if (warp == 1) {
        // ===== MMA issuer: a converged warp whose lane 0 issues; tiles alternate on the pipe =====
        // The warp never touches an mbarrier inside the KV loop: the observer warp (warp 2)
        // waits for every load and P barrier the next MMAs need and meets this warp at the
        // hand-off named barrier. A shared-memory access by the issuing thread behind queued
        // MMAs costs it more than an MMA's shadow (the MMAs' operand reads keep shared memory
        // busy); a named barrier is a hardware barrier and touches no shared memory.
        const uint32_t lead = (lane == 0) ? 1u : 0u;
        bool ok = true;
        for (int g = 0; g < ng && ok; ++g)
            if (!mbar_wait(smem_u32(&bars->q_ready[g]), 0, lim, abort)) {
                if (lane == 0) report(p.status, abort, 1, -1 - g);
                ok = false;
            }
        ok = __all_sync(0xffffffffu, ok);
        // after an error no MMA is issued, but every hand-off still takes place: the
        // observer and this warp always pass the same number of barriers
        const uint32_t iss = ok ? lead : 0u;
        tc_fence_after();
        // tcgen05.mma issue blocks until the tensor pipe has (nearly) drained the previous
        // MMA, so every instruction between MMAs is tensor idle time: the descriptors are
        // precomputed and advanced by constant adds (a descriptor is linear in its 16-byte
        // start address; addresses stay below 256 KB, no carry).
        const uint64_t dq0 = sdesc_sw128(sQ, 16, 1024);
        const uint64_t dk0 = sdesc_sw128(sKV, 16, 1024);
        const uint64_t dv0 = sdesc_sw128(sKV, kBN * 128, 1024);
        // one hand-off: the observer has seen the next awaited barrier complete (or gave up
        // and raised the abort flag; the MMAs then compute on stale operands, which the
        // error status marks as void)
        auto handoff = [&]() {
            named_bar_sync(kBarHandoff, 64);
            tc_fence_after();
        };
        // P_g(j) written to TMEM by softmax group g (its 128 threads arrive)
        auto take_p = [&](int g) {
            named_bar_sync(kBarP + g, 160);
            tc_fence_after();
        };
        // MMA groups: S_g = Q_g K^T (8 MMAs over D) and O_g += P_g V (8 MMAs over the KV
        // tile). `mid(k)` runs after MMA k of a group, in the shadow of the running MMA.
        auto issue_s = [&](int g, int stage, auto&& mid) {
            const uint64_t dq = dq0 + uint64_t((g * C::Q_TILE) >> 4);
            const uint64_t dk = dk0 + uint64_t((stage * C::KV_TILE) >> 4);
            const uint32_t d = tmem + g * kBN;
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {
                const uint64_t off = uint64_t((k >> 2) * ((kBM * 128) >> 4) + (k & 3) * 2);
                umma_ss_if(iss, d, dq + off, dk + off, C::IDESC_S, k > 0 ? 1u : 0u);
                mid(k);
            }
            umma_commit_if(iss, smem_u32(&bars->s_full[g]));
        };
        auto issue_o = [&](int g, int stage, bool acc, auto&& mid) {
            const uint64_t dv = dv0 + uint64_t((stage * C::KV_TILE) >> 4);
            const uint32_t d = tmem + 256 + g * D;
            const uint32_t pa = tmem + g * kBN;   // P_g: bf16 pairs in S_g's columns
#pragma unroll
            for (int k = 0; k < kBN / 16; ++k) {
                umma_ts_if(iss, d, pa + k * 8, dv + uint64_t(k * ((16 * 128) >> 4)), C::IDESC_O,
                           (acc || k > 0) ? 1u : 0u);
                mid(k);
            }
        };
        auto nop = [](int) {};
        // Hand-off sequence (the observer follows the same one): K_0/V_0, then per KV step
        // j the pair K_{j+1}/V_{j+1} (if any); P_g(j) comes straight from group g.
        handoff();
        issue_s(0, 0, nop);
        if (ng == 2) issue_s(1, 0, nop);
        umma_commit_if(iss, smem_u32(&bars->k0_done));
        int sv = 1 % C::STAGES, sk = 2 % C::STAGES;   // ring slots of V_j and K_{j+1}
        for (int j = 0; j < n_tiles; ++j) {
            const bool more = (j + 1) < n_tiles;
            take_p(0);                                  // P_0(j)
            // the release of step j-1 rides in the shadow of PV_0(j)'s second MMA
            issue_o(0, sv, j > 0, [&](int k) {
                if (k == 0 && more) handoff();          // K_{j+1}, V_{j+1}
                if (k == 1 && j > 0) umma_commit_if(iss, smem_u32(&bars->step_done[(j - 1) & 3]));
            });
            if (more) issue_s(0, sk, nop);
            else umma_commit_if(iss, smem_u32(&bars->o_done[0]));
            if (ng == 2) {
                take_p(1);                              // P_1(j)
                issue_o(1, sv, j > 0, nop);
                if (more) issue_s(1, sk, nop);
                else umma_commit_if(iss, smem_u32(&bars->o_done[1]));
            }
            sv = (sv + 2 >= C::STAGES) ? sv + 2 - C::STAGES : sv + 2;
            sk = (sk + 2 >= C::STAGES) ? sk + 2 - C::STAGES : sk + 2;
        }
        // drain: all issued MMAs complete before TMEM is released
        umma_commit_if(lead, smem_u32(&bars->drain[0]));
        mbar_wait_drain(smem_u32(&bars->drain[0]), 0, lim);
      } else if (warp == 2) {
        // ===== observer: waits for what the issuer's next MMAs need, then hands off =====
        // Every wait is bounded; after one gives up (or another role raised the abort flag)
        // the remaining hand-offs pass without waiting, so both warps pass the same number
        // of barriers and the issuer finishes its (void) loop.
        bool ok = true;
        auto observe = [&](uint32_t bar, uint32_t parity, int where) {
            if (ok) {
                ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, lim, abort));
                if (!ok && lane == 0) report(p.status, abort, 4, where);
            }
            named_bar_sync(kBarHandoff, 64);
        };
        // K_j and V_j (loads 2j, 2j+1) complete together on kv_full[j % 4]. Pair j+4 is
        // loaded only after step j-1's slot release, which the issuer commits after this
        // warp saw pair j, so the parity of kv_full[j % 4] is never ambiguous.
        auto kv_bar = [&](int jj) { return smem_u32(&bars->kv_full[jj & 3]); };
        observe(kv_bar(0), 0, 0);
        for (int j = 0; j + 1 < n_tiles; ++j)
            observe(kv_bar(j + 1), ((j + 1) >> 2) & 1, 2 * (j + 1));
      }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsSm));
        // ================================ softmax groups ===============================
        const int g = (warp >> 2) - 1;                 // 0 or 1
        const int sub = warp & 3;                      // TMEM lane quarter of this warp
        const int row = sub * 32 + lane;               // row within the tile
        const int grow = m0 + g * kBM + row;           // query row within the chunk
        const bool active = (g == 0) || active1;
        const uint32_t lane_off = uint32_t(sub * 32) << 16;
        const uint32_t tS = tmem + lane_off + g * kBN;
        const uint32_t tO = tmem + lane_off + 256 + g * D;
        const float sl2 = p.scale_log2;
        bool ok = active;
        if (active) {
            // RoPE-Q: every (cos, sin) of the row is loaded first, while the Q tile's TMA
            // load is still in flight, then the rotation runs once Q has landed. Each
            // entry is one load from an address chosen without branching (the t segment
            // lives in the launch parameters, the h and w segments in the stream's
            // table), so all of them are in flight together; a branch per entry on the
            // runtime segment widths serialises one load latency per entry.
            const bool rot = ROPE && grow < sd.n_q;
            float2 cs[ROPE ? D / 2 : 1];
            if (rot) {
                const int f = grow / p.rope.tpf;
                const int rem = grow - f * p.rope.tpf;
                const int rr = rem / p.rope.gw;
                const int col = rem - rr * p.rope.gw;
                const int dt2 = p.rope.dt2, dth = p.rope.dt2 + p.rope.dh2;
                const float2* t_row = p.rope.t_tab + f * dt2;
                const float2* h_row = p.rope.hw + rr * p.rope.dh2 - dt2;
                const float2* w_row = p.rope.hw + p.rope.gh * p.rope.dh2 + col * p.rope.dw2 - dth;
#pragma unroll
                for (int i = 0; i < (ROPE ? D / 2 : 0); ++i) {
                    const float2* src = i < dt2 ? t_row + i : (i < dth ? h_row + i : w_row + i);
                    cs[i] = *src;
                }
            }
            ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars->q_full), 0, lim, abort));
            if (!ok) report(p.status, abort, 2 + g, -1);
            if (ROPE && ok && rot) {
                uint8_t* qrow = smem + C::OFF_Q + g * C::Q_TILE + row * 128;
#pragma unroll
                for (int c = 0; c < D / 8; ++c) {
                    const int cb = c >> 3, cc = c & 7;
                    uint4* ptr = reinterpret_cast<uint4*>(qrow + cb * (kBM * 128) +
                                                          ((cc ^ (row & 7)) << 4));
                    uint4 v = *ptr;
                    v.x = rope_pair(v.x, cs[4 * c + 0].x, cs[4 * c + 0].y);
                    v.y = rope_pair(v.y, cs[4 * c + 1].x, cs[4 * c + 1].y);
                    v.z = rope_pair(v.z, cs[4 * c + 2].x, cs[4 * c + 2].y);
                    v.w = rope_pair(v.w, cs[4 * c + 3].x, cs[4 * c + 3].y);
                    *ptr = v;
                }
                fence_proxy_async_smem();
            }
            mbar_arrive(smem_u32(&bars->q_ready[g]));
        }
        float m_run = -INFINITY;
        float l_run = 0.0f;
        // Every step ends with this group meeting the MMA warp at its P barrier (named
        // barrier 5 + g: these 128 threads and the MMA warp's 32): the MMA warp waits on it
        // in hardware, no mbarrier and no observer in between. Both sides pass it once per
        // KV step whatever happens: after an error the group keeps passing without
        // computing (a bar.sync, not an arrive, so it can never run a phase ahead). A group
        // with no rows (the second tile of a one-tile item) takes no part: the MMA warp does
        // not issue for it.
        const int p_steps = active ? n_tiles : 0;
        for (int j = 0; j < p_steps; ++j) {
          if (ok) {
            ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars->s_full[g]), j & 1, lim, abort));
            if (!ok) report(p.status, abort, 2 + g, j);
          }
          if (ok) {
            tc_fence_after();
            float s[kBN];
            {
                // the row's 128 scores in one load: one wait instead of four in flight
                uint32_t r[kBN];
                tmem_ld128(tS, r);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < kBN; ++i) s[i] = __uint_as_float(r[i]);
            }
            if (t0 + j == tiles_total - 1) {
                const int valid = sd.n_kv - (t0 + j) * kBN;
#pragma unroll
                for (int i = 0; i < kBN; ++i)
                    if (i >= valid) s[i] = -INFINITY;
            }
            // p = 2^(s * scale * log2 e - m) against a reference m that is the exact row
            // max only on the first tile; afterwards it is left stale. bf16 P shares
            // fp32's exponent range, so stale values are harmless until a p could
            // overflow: every p is bounded by the row sum, so a row sum above
            // kOverflowGuard (rare) triggers the exact max, a rescale of O and a redo.
            // No row-max reduction runs on the common path.
            const uint64_t sl2x2 = f2_pack(sl2, sl2);
            uint32_t pk[32];
            uint64_t acc[4];
            auto exp_half = [&](int h, float mref) {
                const uint64_t negm = f2_pack(-mref, -mref);
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const int e = h * 64 + 2 * i;
                    float x0, x1;
                    f2_unpack(f2_fma(f2_pack(s[e], s[e + 1]), sl2x2, negm), x0, x1);
                    const float p0 = ex2_approx(x0);
                    const float p1 = ex2_approx(x1);
                    acc[i & 3] = f2_add(acc[i & 3], f2_pack(p0, p1));
                    pk[i] = pack_bf16x2(p0, p1);
                }
            };
            auto exp_row = [&](float mref) {
                acc[0] = acc[1] = acc[2] = acc[3] = 0;
                exp_half(0, mref);
                tmem_st32(tS, pk);
                exp_half(1, mref);
                tmem_st32(tS + 32, pk);
            };
            auto row_max = [&]() -> float {   // 8 independent 3-input max chains
                float mx[8];
#pragma unroll
                for (int a = 0; a < 8; ++a) mx[a] = fmaxf(s[a], s[a + 8]);
#pragma unroll
                for (int i = 16; i < kBN; i += 16)
#pragma unroll
                    for (int a = 0; a < 8; ++a) mx[a] = max3f(mx[a], s[i + a], s[i + 8 + a]);
                return max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[5]),
                             fmaxf(mx[6], mx[7]));
            };
            auto row_sum = [&]() -> float {
                float a0, a1, b0, b1, c0, c1, d0, d1;
                f2_unpack(acc[0], a0, a1);
                f2_unpack(acc[1], b0, b1);
                f2_unpack(acc[2], c0, c1);
                f2_unpack(acc[3], d0, d1);
                return ((a0 + a1) + (b0 + b1)) + ((c0 + c1) + (d0 + d1));
            };
            float alpha = 1.0f;
            if (j == 0) {
                m_run = row_max() * sl2;
                exp_row(m_run);
            } else {
                exp_row(m_run);
                const bool big = row_sum() > kOverflowGuard;
                if (__any_sync(0xffffffffu, big)) {
                    const float m_new = fmaxf(m_run, row_max() * sl2);
                    alpha = ex2_approx(m_run - m_new);
                    m_run = m_new;
                    // S_g(j) has landed, so PV_g(j-1) is complete: O_g is stable
#pragma unroll 1
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        tmem_ld32(tO + c * 32, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 32; i += 2) {
                            uint64_t v = f2_mul(
                                f2_pack(__uint_as_float(o[i]), __uint_as_float(o[i + 1])),
                                f2_pack(alpha, alpha));
                            float lo, hi;
                            f2_unpack(v, lo, hi);
                            o[i] = __float_as_uint(lo);
                            o[i + 1] = __float_as_uint(hi);
                        }
                        tmem_st32(tO + c * 32, o);
                    }
                    tmem_st_wait();   // the first P stores complete before they are replaced
                    exp_row(m_run);
                }
            }
            l_run = l_run * alpha + row_sum();
            tmem_st_wait();
            tc_fence_before();
          }
          named_bar_sync(kBarP + g, 160);
        }
        // ---- epilogue ------------------------------------------------------------------
        // O leaves through shared memory and TMA tensor stores. Once both tiles' last PV
        // has completed the K/V ring is free: group g stages its 128-row tile in ring
        // bytes [g * 512 * D, (g + 1) * 512 * D) as blocks of 128 rows x 128 bytes (32 fp32
        // or 64 bf16 columns), 128-byte swizzled (16-byte chunk i of row r sits at chunk
        // i ^ (r & 7)), which is the layout the tensor maps read. Rows past Nq are clipped
        // by the store.
        if (ok) {
            bool got = mbar_wait(smem_u32(&bars->o_done[g]), 0, lim, abort);
            if (got && ng == 2) got = mbar_wait(smem_u32(&bars->o_done[1 - g]), 0, lim, abort);
            ok = __all_sync(0xffffffffu, got);
            if (!ok) report(p.status, abort, 2 + g, 4000);
        }
        const uint32_t stg = sKV + uint32_t(g * 512 * D);
        const uint32_t sw = uint32_t(row & 7);
        const bool leader = (sub == 0) && (lane == 0);    // issues the group's TMA copies
        auto stage_f32 = [&](int c, const float (&v)[32]) {   // columns [32c, 32c + 32)
            const uint32_t rb = stg + uint32_t(c * 16384 + row * 128);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                st_shared_v4(rb + ((uint32_t(i) ^ sw) << 4), __float_as_uint(v[4 * i]),
                             __float_as_uint(v[4 * i + 1]), __float_as_uint(v[4 * i + 2]),
                             __float_as_uint(v[4 * i + 3]));
        };
        auto stage_bf16 = [&](int c, const float (&v)[32]) {  // columns [32c, 32c + 32)
            const uint32_t rb = stg + uint32_t((c >> 1) * 16384 + row * 128);
#pragma unroll
            for (int i = 0; i < 4; ++i)
                st_shared_v4(rb + ((uint32_t((c & 1) * 4 + i) ^ sw) << 4),
                             pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                             pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
        };
        // staged tile -> out (the group's leader); the CTA may exit once the reads are done
        auto store_out = [&]() {
            fence_proxy_async_smem();
            named_bar_sync(2 + g, 128);
            if (ok && leader) {
                const int nb = p.out_bf16 ? D / 64 : D / 32;
                for (int cb = 0; cb < nb; ++cb)
                    tma_store_3d(&sd.out_map, stg + uint32_t(cb * 16384), cb * (p.out_bf16 ? 64 : 32),
                                 head, m0 + g * kBM);
                bulk_commit();
                bulk_wait_read<0>();
            }
        };
        // the item's split coordinates, re-derived from the block index here instead of
        // kept live through the KV loop (registers are scarce in the softmax warps: kept
        // live, they made the compiler spill inside the fused RoPE variant)
        int e_split = 0, e_parts = 1, e_tail = 0;
        {
            int cid;
            asm volatile("mov.u32 %0, %%ctaid.x;" : "=r"(cid));
            if (cid >= p.n_full) {
                const int v = cid - p.n_full;
                e_tail = v / p.n_split;
                e_split = v - e_tail * p.n_split;
                e_parts = p.n_split;
            }
        }
        if (e_parts == 1) {
            if (ok) {
                // O / l -> out
                tc_fence_after();
                const float inv_l = 1.0f / l_run;
#pragma unroll 1
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(tO + c * 32, o);
                    tmem_ld_wait();
                    float v[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(o[i]) * inv_l;
                    if (p.out_bf16) stage_bf16(c, v);
                    else stage_f32(c, v);
                }
            }
            store_out();
        } else {
            // unnormalised partial of this split -> scratch (rows of tile (tail group, split, g))
            const int prow_tile = int((size_t(e_tail) * e_parts + e_split) * 2 * kBM) + g * kBM;
            if (ok) {
                tc_fence_after();
#pragma unroll 1
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(tO + c * 32, o);
                    tmem_ld_wait();
                    float v[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(o[i]);
                    stage_f32(c, v);
                }
                p.part_ml[prow_tile + row] = make_float2(m_run, l_run);
            }
            fence_proxy_async_smem();
            named_bar_sync(2 + g, 128);
            if (ok && leader) {
                for (int cb = 0; cb < D / 32; ++cb)
                    tma_store_2d(&p.part_map, stg + uint32_t(cb * 16384), cb * 32, prow_tile);
                bulk_commit();
                bulk_wait<0>();   // written, not only read: other CTAs read it next
                fence_proxy_async_global();
            }
            __threadfence();
            // the last split of this query group to finish merges all partials
            named_bar_sync(1, 256);
            if (threadIdx.x == 128) {
                const int old = atomicAdd(p.counters + e_tail, 1);
                const int last = (old == e_parts - 1);
                if (last) p.counters[e_tail] = 0;    // every split has counted: reset for reuse
                bars->last_split = last;
            }
            named_bar_sync(1, 256);
            if (bars->last_split) {
                __threadfence();
                fence_proxy_async_global();
                const int prow0 = int(size_t(e_tail) * e_parts * 2 * kBM) + g * kBM;
                float2 ml[kMaxSplit];
#pragma unroll
                for (int r = 0; r < kMaxSplit; ++r)
                    ml[r] = (r == e_split) ? make_float2(m_run, l_run)
                            : (r < e_parts) ? __ldcg(&p.part_ml[prow0 + r * 2 * kBM + row])
                                              : make_float2(-INFINITY, 0.0f);
                float mref = -INFINITY;
#pragma unroll
                for (int r = 0; r < kMaxSplit; ++r) mref = fmaxf(mref, ml[r].x);
                float wr[kMaxSplit];
                float lsum = 0.0f;
#pragma unroll
                for (int r = 0; r < kMaxSplit; ++r) {
                    wr[r] = (r < e_parts) ? ex2_approx(ml[r].x - mref) : 0.0f;
                    lsum += wr[r] * ml[r].y;
                }
                const float w_own = ex2_approx(m_run - mref);
                // splits are accumulated in index order whichever of them merges, so the
                // result does not depend on which split finished last: this split's own O
                // comes from TMEM, the others' tiles through the group's staging, and the
                // running sum lives in the group's S columns of TMEM (free by now)
                const uint32_t tAcc = tS;
                bool first = true;
                int phase = 0;
#pragma unroll
                for (int r = 0; r < kMaxSplit; ++r) {
                    if (r >= e_parts) continue;
                    const bool own = (r == e_split);
                    if (!own) {
                        const uint32_t fb = smem_u32(&bars->epi_full[g]);
                        if (ok && leader) {
                            mbar_arrive_expect_tx(fb, uint32_t(512 * D));
                            for (int cb = 0; cb < D / 32; ++cb)
                                tma_load_2d(stg + uint32_t(cb * 16384), &p.part_map, fb, cb * 32,
                                            prow0 + r * 2 * kBM);
                        }
                        bool got = ok;
                        if (got) {
                            // the leader drains its own load even after an abort elsewhere
                            got = leader ? mbar_wait_drain(fb, phase & 1, lim)
                                         : mbar_wait(fb, phase & 1, lim, abort);
                            got = __all_sync(0xffffffffu, got);
                            if (!got) report(p.status, abort, 2 + g, 5000 + r);
                        }
                        ok = ok && got;
                        ++phase;
                    }
                    if (ok) {
                        const float w = own ? w_own : wr[r];
                        tc_fence_after();
#pragma unroll 1
                        for (int c = 0; c < D / 32; ++c) {
                            float x[32];
                            if (own) {
                                uint32_t o[32];
                                tmem_ld32(tO + c * 32, o);
                                tmem_ld_wait();
#pragma unroll
                                for (int i = 0; i < 32; ++i) x[i] = __uint_as_float(o[i]);
                            } else {
                                const uint32_t rb = stg + uint32_t(c * 16384 + row * 128);
#pragma unroll
                                for (int i = 0; i < 8; ++i) {
                                    const uint4 q4 = ld_shared_v4(rb + ((uint32_t(i) ^ sw) << 4));
                                    x[4 * i] = __uint_as_float(q4.x);
                                    x[4 * i + 1] = __uint_as_float(q4.y);
                                    x[4 * i + 2] = __uint_as_float(q4.z);
                                    x[4 * i + 3] = __uint_as_float(q4.w);
                                }
                            }
                            uint32_t a[32];
                            if (first) {
#pragma unroll
                                for (int i = 0; i < 32; ++i) a[i] = __float_as_uint(0.0f + w * x[i]);
                            } else {
                                tmem_ld32(tAcc + c * 32, a);
                                tmem_ld_wait();
#pragma unroll
                                for (int i = 0; i < 32; ++i)
                                    a[i] = __float_as_uint(__uint_as_float(a[i]) + w * x[i]);
                            }
                            tmem_st32(tAcc + c * 32, a);
                        }
                        tmem_st_wait();
                        tc_fence_before();
                    }
                    first = false;
                    if (!own) named_bar_sync(2 + g, 128);   // staging is refilled next
                }
                if (ok) {
                    const float inv_l = 1.0f / lsum;
                    tc_fence_after();
#pragma unroll 1
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t a[32];
                        tmem_ld32(tAcc + c * 32, a);
                        tmem_ld_wait();
                        float x[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) x[i] = __uint_as_float(a[i]) * inv_l;
                        if (p.out_bf16) stage_bf16(c, x);
                        else stage_f32(c, x);
                    }
                }
                store_out();
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, 512);
}

template <int D, int MAXS, bool ROPE>
cudaError_t launch(const AttnParams<MAXS>& p, cudaStream_t st) {
    if (p.total_items <= 0) return cudaSuccess;
    auto kern = attn_kernel<D, MAXS, ROPE>;
    static bool attr_set[kMaxDevices] = {};   // per device: attributes are per device
    const int dev = device_slot();
    if (dev < 0 || !attr_set[dev]) {
        // the setmaxnreg split assumes exactly kRegsLaunch registers per thread at launch;
        // any other allocation could leave the increase waiting, so refuse to launch
        cudaFuncAttributes fa;
        cudaError_t e = cudaFuncGetAttributes(&fa, kern);
        if (e != cudaSuccess) return e;
        if (fa.numRegs != kRegsLaunch) return cudaErrorInvalidConfiguration;
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 Cfg<D>::SMEM);
        if (e != cudaSuccess) return e;
        if (dev >= 0) attr_set[dev] = true;
    }
    kern<<<p.total_items, kThreads, Cfg<D>::SMEM, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attention_single(const AttnParams<1>& p, int head_dim, bool rope_q,
                                    cudaStream_t st) {
    if (head_dim == 128)
        return rope_q ? launch<128, 1, true>(p, st) : launch<128, 1, false>(p, st);
    if (head_dim == 64)
        return rope_q ? launch<64, 1, true>(p, st) : launch<64, 1, false>(p, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_attention_batched(const AttnParams<kMaxBatchStreams>& p, int head_dim,
                                     cudaStream_t st) {
    if (head_dim == 128) return launch<128, kMaxBatchStreams, false>(p, st);
    if (head_dim == 64) return launch<64, kMaxBatchStreams, false>(p, st);
    return cudaErrorInvalidValue;
}

}  // namespace frt
