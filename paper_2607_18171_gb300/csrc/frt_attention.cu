// frt_attention.cu — chunk flash attention over the rolling KV cache on sm_103a.
//
// out[i,h,:] = sum_j softmax_j(scale * <q_i, k_j>) v_j over every valid cache row j
// (the whole window is visible to every query of the chunk: bidirectional within the
// chunk, all earlier chunks of the window), bf16 operands, fp32 accumulation.
//
// One CTA = one work item = (stream, head, 256 query rows as two 128-row tiles).
// Warp roles (320 threads, one CTA per SM):
//   warp 0      TMA producer: Q tiles once, then K/V tiles through a STAGES-deep ring
//               in the order the MMA consumes them (K0, K1, V0, K2, V1, ...).
//   warp 1      TMEM allocator + single-thread tcgen05.mma issuer:
//                 S_g = Q_g K_j^T  (M=128, N=128, K=D; fp32 in TMEM)
//                 O_g += P_g V_j   (M=128, N=D,   K=128; fp32 in TMEM)
//   warps 2-5   softmax group 0 (query tile 0), one thread per query row
//   warps 6-9   softmax group 1 (query tile 1)
// TMEM (512 columns): S_0 [0,128), S_1 [128,256), O_0 [256,256+D), O_1 [256+D,256+2D).
// The softmax threads read S with tcgen05.ld, keep a running max in the log2 domain,
// write P (bf16) to shared memory in the 128-byte-swizzled K-major layout the MMA
// reads, and rescale O in TMEM only when the running max grows by more than
// 2^kRescaleLog2 (O and the row sum stay consistently scaled, so the result is exact).
//
// Every wait is bounded (mbar_wait): a role that gives up records FRT_ERR_TIMEOUT in the
// stream's status block, raises a CTA-wide abort flag, and the CTA drains its in-flight
// TMA/MMA work (bounded) and frees TMEM before exiting.
#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {

namespace {

constexpr int kThreads = 320;
constexpr int kBM = 128;   // query rows per tile
constexpr int kBN = 128;   // KV rows per tile
constexpr float kRescaleLog2 = 8.0f;
constexpr int kTimeoutCode = 6;  // FRT_ERR_TIMEOUT

template <int D>
struct Cfg {
    static constexpr int NCB = D / 64;                 // 128-byte column blocks per row
    static constexpr int Q_TILE = kBM * D * 2;
    static constexpr int KV_TILE = kBN * D * 2;
    static constexpr int P_TILE = kBM * kBN * 2;
    static constexpr int STAGES = (D == 128) ? 3 : 6;
    static constexpr int OFF_Q = 0;
    static constexpr int OFF_P = OFF_Q + 2 * Q_TILE;
    static constexpr int OFF_KV = OFF_P + 2 * P_TILE;
    static constexpr int OFF_BAR = OFF_KV + STAGES * KV_TILE;
    static constexpr int SMEM = OFF_BAR + 256 + 1024;  // barriers + alignment slack
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(kBM, kBN, false);
    static constexpr uint32_t IDESC_O = idesc_bf16_f32(kBM, D, true);
};

struct Bars {
    uint64_t q_full;
    uint64_t q_ready[2];
    uint64_t s_full[2];
    uint64_t s_free[2];
    uint64_t p_full[2];
    uint64_t o_done[2];
    uint64_t drain;
    uint64_t kv_full[8];
    uint64_t kv_empty[8];
    uint32_t tmem_base;
    int abort_flag;
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

// Position of KV load number L in the consumption order K0, K1, V0, K2, V1, ...
// Returns the tile index and whether it is a V tile.
__device__ __forceinline__ void kv_load_at(int L, int n_tiles, int& tile, bool& is_v) {
    if (L == 0) { tile = 0; is_v = false; return; }
    // after K0: pairs (K_{t}, V_{t-1}) for t = 1..n-1, then V_{n-1}
    const int t = (L + 1) >> 1;            // L=1 -> t=1 (K1), L=2 -> t=1 (V0) ...
    if (t < n_tiles) {
        if (L & 1) { tile = t; is_v = false; }
        else       { tile = t - 1; is_v = true; }
    } else {
        tile = n_tiles - 1; is_v = true;   // L = 2n-1
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
    const uint32_t sP = smem_u32(smem + C::OFF_P);
    const uint32_t sKV = smem_u32(smem + C::OFF_KV);
    volatile int* abort = &bars->abort_flag;

    // ---- work item ---------------------------------------------------------------------
    const int item = blockIdx.x;
    int si = 0;
    while (si + 1 < p.n_streams && item >= p.s[si + 1].item_begin) ++si;
    const AttnStreamDesc& sd = p.s[si];
    const int local = item - sd.item_begin;
    const int head = local / sd.n_qpairs;
    const int m0 = (local - head * sd.n_qpairs) * (2 * kBM);
    const bool active1 = (m0 + kBM) < sd.n_q;
    const int n_tiles = (sd.n_kv + kBN - 1) / kBN;
    const int n_loads = 2 * n_tiles;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bars->q_full), 1);
        for (int g = 0; g < 2; ++g) {
            mbar_init(smem_u32(&bars->q_ready[g]), kBM);
            mbar_init(smem_u32(&bars->s_full[g]), 1);
            mbar_init(smem_u32(&bars->s_free[g]), kBM);
            mbar_init(smem_u32(&bars->p_full[g]), kBM);
            mbar_init(smem_u32(&bars->o_done[g]), 1);
        }
        mbar_init(smem_u32(&bars->drain), 1);
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(smem_u32(&bars->kv_full[s]), 1);
            mbar_init(smem_u32(&bars->kv_empty[s]), 1);
        }
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

    if (warp == 0) {
        // ================================ TMA producer =================================
        if (lane == 0) {
            tma_prefetch_map(&sd.q_map);
            tma_prefetch_map(&sd.k_map);
            tma_prefetch_map(&sd.v_map);
            const uint32_t qbar = smem_u32(&bars->q_full);
            mbar_arrive_expect_tx(qbar, (active1 ? 2 : 1) * C::Q_TILE);
            for (int g = 0; g < (active1 ? 2 : 1); ++g)
                for (int cb = 0; cb < C::NCB; ++cb)
                    tma_load_3d(sQ + g * C::Q_TILE + cb * (kBM * 128), &sd.q_map, qbar,
                                cb * 64, head, m0 + g * kBM);
            int L = 0;
            for (; L < n_loads; ++L) {
                const int stage = L % C::STAGES;
                const int round = L / C::STAGES;
                if (round > 0 &&
                    !mbar_wait(smem_u32(&bars->kv_empty[stage]), (round - 1) & 1, lim, abort)) {
                    report(p.status, abort, 0, L);
                    break;
                }
                int tile; bool is_v;
                kv_load_at(L, n_tiles, tile, is_v);
                const CUtensorMap* map = is_v ? &sd.v_map : &sd.k_map;
                const uint32_t fb = smem_u32(&bars->kv_full[stage]);
                mbar_arrive_expect_tx(fb, C::KV_TILE);
                const uint32_t dst = sKV + stage * C::KV_TILE;
                for (int cb = 0; cb < C::NCB; ++cb)
                    tma_load_3d(dst + cb * (kBN * 128), map, fb, cb * 64, head, tile * kBN);
            }
            // drain: every issued load must have landed before the CTA may exit
            const int first = (L - C::STAGES) > 0 ? (L - C::STAGES) : 0;
            for (int Ld = first; Ld < L; ++Ld)
                mbar_wait(smem_u32(&bars->kv_full[Ld % C::STAGES]), (Ld / C::STAGES) & 1,
                          lim, abort);
            mbar_wait(qbar, 0, lim, abort);
        }
    } else if (warp == 1) {
        // ================================ MMA issuer ===================================
        if (lane == 0) {
            bool ok = true;
            const int ng = active1 ? 2 : 1;
            for (int g = 0; g < ng && ok; ++g)
                if (!mbar_wait(smem_u32(&bars->q_ready[g]), 0, lim, abort)) {
                    report(p.status, abort, 1, -1 - g);
                    ok = false;
                }
            tc_fence_after();
            int L = 0;
            auto wait_load = [&](int Lw) -> bool {
                if (!mbar_wait(smem_u32(&bars->kv_full[Lw % C::STAGES]), (Lw / C::STAGES) & 1,
                               lim, abort)) {
                    report(p.status, abort, 1, Lw);
                    return false;
                }
                tc_fence_after();
                return true;
            };
            auto issue_s = [&](int g, int stage) {
                const uint32_t d = tmem + g * kBN;
                const uint32_t qa = sQ + g * C::Q_TILE;
                const uint32_t kb = sKV + stage * C::KV_TILE;
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    const uint32_t off = (k >> 2) * (kBM * 128) + (k & 3) * 32;
                    umma_ss(d, sdesc_sw128(qa + off, 16, 1024), sdesc_sw128(kb + off, 16, 1024),
                            C::IDESC_S, k > 0 ? 1u : 0u);
                }
                umma_commit(smem_u32(&bars->s_full[g]));
            };
            auto issue_o = [&](int g, int stage, bool acc) {
                const uint32_t d = tmem + 256 + g * D;
                const uint32_t pa = sP + g * C::P_TILE;
                const uint32_t vb = sKV + stage * C::KV_TILE;
#pragma unroll
                for (int k = 0; k < kBN / 16; ++k) {
                    const uint32_t aoff = (k >> 2) * (kBM * 128) + (k & 3) * 32;
                    const uint32_t boff = k * (16 * 128);
                    umma_ss(d, sdesc_sw128(pa + aoff, 16, 1024),
                            sdesc_sw128(vb + boff, kBN * 128, 1024), C::IDESC_O,
                            (acc || k > 0) ? 1u : 0u);
                }
                umma_commit(smem_u32(&bars->o_done[g]));
            };
            if (ok && (ok = wait_load(L))) {
                const int k0 = L % C::STAGES;
                for (int g = 0; g < ng; ++g) issue_s(g, k0);
                umma_commit(smem_u32(&bars->kv_empty[k0]));
                ++L;
            }
            for (int j = 0; j < n_tiles && ok; ++j) {
                const bool more = (j + 1) < n_tiles;
                int kst = -1, vst;
                if (more) {
                    if (!(ok = wait_load(L))) break;
                    kst = L % C::STAGES;
                    ++L;
                }
                if (!(ok = wait_load(L))) break;
                vst = L % C::STAGES;
                ++L;
                for (int g = 0; g < ng && ok; ++g) {
                    if (more) {
                        if (!mbar_wait(smem_u32(&bars->s_free[g]), j & 1, lim, abort)) {
                            report(p.status, abort, 1, 1000 + j);
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        issue_s(g, kst);
                    }
                    if (!mbar_wait(smem_u32(&bars->p_full[g]), j & 1, lim, abort)) {
                        report(p.status, abort, 1, 2000 + j);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    issue_o(g, vst, j > 0);
                }
                if (!ok) break;
                if (more) umma_commit(smem_u32(&bars->kv_empty[kst]));
                umma_commit(smem_u32(&bars->kv_empty[vst]));
            }
            // drain: all issued MMAs complete before TMEM is released
            umma_commit(smem_u32(&bars->drain));
            mbar_wait(smem_u32(&bars->drain), 0, lim, abort);
        }
    } else {
        // ================================ softmax groups ===============================
        const int g = (warp - 2) >> 2;                 // 0 or 1
        const int sub = warp & 3;                      // TMEM lane quarter of this warp
        const int row = sub * 32 + lane;               // row within the tile
        const int grow = m0 + g * kBM + row;           // query row within the chunk
        const bool active = (g == 0) || active1;
        const uint32_t lane_off = uint32_t(sub * 32) << 16;
        const uint32_t tS = tmem + lane_off + g * kBN;
        const uint32_t tO = tmem + lane_off + 256 + g * D;
        const uint32_t pRow = sP + g * C::P_TILE + row * 128;
        const float sl2 = p.scale_log2;
        bool ok = active;
        if (active) {
            if (!mbar_wait(smem_u32(&bars->q_full), 0, lim, abort)) {
                report(p.status, abort, 2 + g, -1);
                ok = false;
            }
            if (ROPE && ok && grow < sd.n_q) {
                const int f = grow / p.rope.tpf;
                const int rem = grow - f * p.rope.tpf;
                const int rr = rem / p.rope.gw;
                const int col = rem - rr * p.rope.gw;
                uint8_t* qrow = smem + C::OFF_Q + g * C::Q_TILE + row * 128;
#pragma unroll
                for (int c = 0; c < D / 8; ++c) {
                    const int cb = c >> 3, cc = c & 7;
                    uint4* ptr = reinterpret_cast<uint4*>(qrow + cb * (kBM * 128) +
                                                          ((cc ^ (row & 7)) << 4));
                    *ptr = rope_rotate8(*ptr, c * 8, f, rr, col, p.rope);
                }
                fence_proxy_async_smem();
            }
            mbar_arrive(smem_u32(&bars->q_ready[g]));
        }
        float m_run = -INFINITY;
        float l_run = 0.0f;
        for (int j = 0; j < n_tiles && ok; ++j) {
            if (!mbar_wait(smem_u32(&bars->s_full[g]), j & 1, lim, abort)) {
                report(p.status, abort, 2 + g, j);
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t sr[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(tS + c * 32, sr[c]);
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(smem_u32(&bars->s_free[g]));

            float s[kBN];
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(sr[c][i]);
            if (j == n_tiles - 1) {
                const int valid = sd.n_kv - j * kBN;
#pragma unroll
                for (int i = 0; i < kBN; ++i)
                    if (i >= valid) s[i] = -INFINITY;
            }
            float mx = s[0];
#pragma unroll
            for (int i = 1; i < kBN; ++i) mx = fmaxf(mx, s[i]);
            const float m_new = fmaxf(m_run, mx * sl2);
            const bool need = m_new > m_run + kRescaleLog2;
            float alpha = 1.0f;
            if (need) {
                alpha = ex2_approx(m_run - m_new);
                m_run = m_new;
            }
            const float neg_m = -m_run;
            float rs = 0.0f;
            uint32_t pk[kBN / 2];
#pragma unroll
            for (int i = 0; i < kBN; i += 2) {
                const float p0 = ex2_approx(__fmaf_rn(s[i], sl2, neg_m));
                const float p1 = ex2_approx(__fmaf_rn(s[i + 1], sl2, neg_m));
                rs += p0 + p1;
                pk[i >> 1] = pack_bf16x2(p0, p1);
            }
            l_run = l_run * alpha + rs;

            if (j > 0) {
                // PV of the previous tile must be done: P buffer reuse and O rescale
                if (!mbar_wait(smem_u32(&bars->o_done[g]), (j - 1) & 1, lim, abort)) {
                    report(p.status, abort, 2 + g, 3000 + j);
                    ok = false;
                    break;
                }
                tc_fence_after();
            }
            // P row -> shared memory, K-major 128-byte swizzle (16-byte chunk c of a
            // 128-byte row lives at chunk position c ^ (row % 8))
#pragma unroll
            for (int c = 0; c < kBN / 8; ++c) {
                const int cb = c >> 3, cc = c & 7;
                const uint32_t addr = pRow + cb * (kBM * 128) + ((cc ^ (row & 7)) << 4);
                asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr),
                             "r"(pk[4 * c]), "r"(pk[4 * c + 1]), "r"(pk[4 * c + 2]),
                             "r"(pk[4 * c + 3])
                             : "memory");
            }
            if (j > 0 && __any_sync(0xffffffffu, need)) {
#pragma unroll 1
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(tO + c * 32, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                    tmem_st32(tO + c * 32, o);
                }
                tmem_st_wait();
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(smem_u32(&bars->p_full[g]));
        }
        // ---- epilogue: O / l -> global -------------------------------------------------
        if (ok) {
            if (!mbar_wait(smem_u32(&bars->o_done[g]), (n_tiles - 1) & 1, lim, abort)) {
                report(p.status, abort, 2 + g, 4000);
                ok = false;
            }
        }
        if (ok) {
            tc_fence_after();
            const float inv_l = 1.0f / l_run;
            const bool store = grow < sd.n_q;
            const size_t obase = (size_t(grow) * p.heads + head) * D;
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                tmem_ld32(tO + c * 32, o);
                tmem_ld_wait();
                if (store) {
                    if (p.out_bf16) {
                        uint4* dst = reinterpret_cast<uint4*>(
                            static_cast<uint16_t*>(sd.out) + obase + c * 32);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            uint4 w;
                            w.x = pack_bf16x2(__uint_as_float(o[8 * i + 0]) * inv_l,
                                              __uint_as_float(o[8 * i + 1]) * inv_l);
                            w.y = pack_bf16x2(__uint_as_float(o[8 * i + 2]) * inv_l,
                                              __uint_as_float(o[8 * i + 3]) * inv_l);
                            w.z = pack_bf16x2(__uint_as_float(o[8 * i + 4]) * inv_l,
                                              __uint_as_float(o[8 * i + 5]) * inv_l);
                            w.w = pack_bf16x2(__uint_as_float(o[8 * i + 6]) * inv_l,
                                              __uint_as_float(o[8 * i + 7]) * inv_l);
                            dst[i] = w;
                        }
                    } else {
                        float4* dst = reinterpret_cast<float4*>(
                            static_cast<float*>(sd.out) + obase + c * 32);
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            dst[i] = make_float4(__uint_as_float(o[4 * i + 0]) * inv_l,
                                                 __uint_as_float(o[4 * i + 1]) * inv_l,
                                                 __uint_as_float(o[4 * i + 2]) * inv_l,
                                                 __uint_as_float(o[4 * i + 3]) * inv_l);
                    }
                }
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
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             Cfg<D>::SMEM);
        if (e != cudaSuccess) return e;
        attr_set = true;
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
