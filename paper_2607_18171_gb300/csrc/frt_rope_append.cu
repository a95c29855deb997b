// frt_rope_append.cu — the two HBM-bound kernels of the path, as one staged kernel:
//   * KV append into the sliding-window ring slot, optionally rotating K on the way
//     (frt_kv_append_evict / the fused frt_chunk_step): A = K (rotated or not), B = V;
//   * 3D RoPE of q and k in place (frt_rope3d_qk): A = q, B = k, both rotated.
// Token rows ([heads * head_dim] bf16, contiguous) move global -> shared -> global with
// bulk copies (cp.async.bulk) through a ring of up to kMaxStages blocks of consecutive
// tokens: one thread drives the copy engine (loads ahead, stores behind), seven warps
// rotate the rows that need it in shared memory. V never passes through registers.
// One CTA per SM keeps up to 200 KB of rows (~40 KB per stage) in flight.
#include <algorithm>

#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {

namespace {
constexpr int kThreads = 256;           // warp 0: copy driver; warps 1-7: rotation
constexpr int kWorkers = kThreads - 32;
constexpr int kMaxStages = 6;
constexpr int kStageTarget = 40 * 1024; // bytes of A + B rows per stage (target)
constexpr int kSmemBudget = 200 * 1024;
constexpr int kTimeoutCode = 6;         // FRT_ERR_TIMEOUT

struct StagedParams {
    const uint8_t* a_src;
    const uint8_t* b_src;
    uint8_t* a_dst;
    uint8_t* b_dst;
    int rot_a, rot_b;        // rotate A / B rows
    int n_tok;
    int row_bytes;           // heads * head_dim * 2
    int vec_per_tok;         // row_bytes / 16
    int vec_per_head_log2;   // log2(head_dim / 8)
    int tok_per_block;       // tokens per stage
    int stages;              // ring depth (<= kMaxStages)
    int coop;                // rotation: all worker warps share each token (wide rows)
    const uint8_t* a_lo;     // destination extents [lo, hi) checked by the FRT_DEBUG build
    const uint8_t* a_hi;
    const uint8_t* b_lo;
    const uint8_t* b_hi;
    unsigned long long wait_limit_ns;
    DeviceStatus* status;
    RopeArgs ra;
};

__device__ __forceinline__ void report(DeviceStatus* st, volatile int* abort, int role, int where) {
    *abort = 1;
    if (st != nullptr) {
        volatile DeviceStatus* s = st;
        if (s->code == 0) {
            s->block = blockIdx.x;
            s->role = 100 + role;
            s->where = where;
            __threadfence_system();
            s->code = kTimeoutCode;
        }
    }
}

__global__ void __launch_bounds__(kThreads, 1) staged_rows_kernel(const __grid_constant__ StagedParams p) {
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ uint64_t full[kMaxStages], done[kMaxStages];
    __shared__ float2 s_t[kMaxTEntries];
    __shared__ int abort_flag;
    volatile int* abort = &abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int T = p.tok_per_block;
    const int kStages = p.stages;
    const uint32_t half = uint32_t(T) * p.row_bytes;       // A (or B) rows of one stage
    const int n_blocks = (p.n_tok + T - 1) / T;
    const int my_n = blockIdx.x < n_blocks ? (n_blocks - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&done[s]), kWorkers);
        }
        abort_flag = 0;
        fence_mbar_init();
    }
    // the chunk's t-segment table: shared memory (lanes index it divergently)
    if (p.rot_a | p.rot_b)
        for (int i = threadIdx.x; i < kMaxTEntries; i += kThreads) s_t[i] = p.ra.t_tab[i];
    __syncthreads();
    const uint32_t ring0 = smem_u32(ring);
    const uint64_t lim = p.wait_limit_ns;

    if (warp == 0) {
        if (lane == 0) {
            int issued = 0, stored = 0;
            auto load = [&](int i) {
                const int s = i % kStages;
                const int tok0 = (blockIdx.x + i * gridDim.x) * T;
                const uint32_t bytes = uint32_t(min(T, p.n_tok - tok0)) * p.row_bytes;
                const uint32_t fb = smem_u32(&full[s]);
                mbar_arrive_expect_tx(fb, 2 * bytes);
                bulk_load(ring0 + s * 2 * half, p.a_src + size_t(tok0) * p.row_bytes, bytes, fb);
                bulk_load(ring0 + s * 2 * half + half, p.b_src + size_t(tok0) * p.row_bytes, bytes, fb);
                ++issued;
            };
            for (int i = 0; i < kStages - 1 && i < my_n; ++i) load(i);
            for (int i = 0; i < my_n; ++i) {
                const int s = i % kStages;
                if (!mbar_wait(smem_u32(&done[s]), (i / kStages) & 1, lim, abort)) {
                    report(p.status, abort, 0, i);
                    break;
                }
                const int tok0 = (blockIdx.x + i * gridDim.x) * T;
                const uint32_t bytes = uint32_t(min(T, p.n_tok - tok0)) * p.row_bytes;
                uint8_t* ad = p.a_dst + size_t(tok0) * p.row_bytes;
                uint8_t* bd = p.b_dst + size_t(tok0) * p.row_bytes;
#ifdef FRT_DEBUG
                // a store outside its destination's extent is recorded and skipped
                if (ad < p.a_lo || ad + bytes > p.a_hi || bd < p.b_lo || bd + bytes > p.b_hi) {
                    record_status(p.status, kStatusBounds, 102, tok0);
                } else
#endif
                {
                    bulk_store(ad, ring0 + s * 2 * half, bytes);
                    bulk_store(bd, ring0 + s * 2 * half + half, bytes);
                }
                bulk_commit();
                ++stored;
                // block i + kStages - 1 reuses the stage of block i - 1: its stores must
                // have finished reading shared memory (all but the newest group)
                if (i + kStages - 1 < my_n) {
                    bulk_wait_read<1>();
                    load(i + kStages - 1);
                }
            }
            // drain: loads issued but never stored (error path) must land before exit
            for (int i = stored; i < issued; ++i)
                mbar_wait_drain(smem_u32(&full[i % kStages]), (i / kStages) & 1, lim);
            bulk_wait_read<0>();
        }
    } else {
        // Narrow rows: one warp per token. Wide rows (p.coop): all seven warps share each
        // token, so a stage of one or two wide tokens does not leave five warps idle. In
        // both a lane's 16-byte vectors all sit at the same head_dim offset (the stride,
        // 32 or 224 vectors, is a multiple of the vectors per head), so its four
        // (cos, sin) pairs are fetched once per token and reused for every head.
        const int wid = warp - 1;
        const int d0 = (lane & ((1 << p.vec_per_head_log2) - 1)) * 8;
        const int t_first = p.coop ? 0 : wid, t_step = p.coop ? 1 : kWorkers / 32;
        const int v_first = p.coop ? wid * 32 + lane : lane, v_step = p.coop ? kWorkers : 32;
        for (int i = 0; i < my_n; ++i) {
            const int s = i % kStages;
            if (!mbar_wait(smem_u32(&full[s]), (i / kStages) & 1, lim, abort)) {
                report(p.status, abort, 1, i);
                break;
            }
            const int tok0 = (blockIdx.x + i * gridDim.x) * T;
            const int nt = min(T, p.n_tok - tok0);
            for (int ab = 0; ab < 2; ++ab) {
                if (!(ab == 0 ? p.rot_a : p.rot_b)) continue;
                uint4* rows = reinterpret_cast<uint4*>(ring + s * 2 * half + ab * half);
                for (int t = t_first; t < nt; t += t_step) {
                    const int tok = tok0 + t;
                    const int f = tok / p.ra.tpf;
                    const int rem = tok - f * p.ra.tpf;
                    const int r = rem / p.ra.gw;
                    const int col = rem - r * p.ra.gw;
                    float2 cs[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) cs[q] = rope_cs(p.ra, s_t, (d0 >> 1) + q, f, r, col);
                    uint4* tr = rows + size_t(t) * p.vec_per_tok;
                    for (int v = v_first; v < p.vec_per_tok; v += v_step) {
                        uint4 x = tr[v];
                        x.x = rope_pair(x.x, cs[0].x, cs[0].y);
                        x.y = rope_pair(x.y, cs[1].x, cs[1].y);
                        x.z = rope_pair(x.z, cs[2].x, cs[2].y);
                        x.w = rope_pair(x.w, cs[3].x, cs[3].y);
                        tr[v] = x;
                    }
                }
            }
            fence_proxy_async_smem();   // rotated rows -> visible to the bulk store
            mbar_arrive(smem_u32(&done[s]));
        }
    }
    __syncthreads();
}

cudaError_t launch_staged(StagedParams& sp, cudaStream_t st) {
    sp.tok_per_block = std::max(1, std::min(sp.n_tok, kStageTarget / (2 * sp.row_bytes)));
    const int stage_bytes = 2 * sp.tok_per_block * sp.row_bytes;
    sp.stages = std::min(kMaxStages, kSmemBudget / stage_bytes);
    // rows of at least two vectors per worker thread are rotated by all worker warps
    // together (measured at 40 heads x 128, 10 KB rows, two tokens per stage: 720p append
    // 5547 -> 6053 GB/s); narrower rows keep one warp per token (3 KB rows measured
    // 3410 -> 2112 GB/s the other way)
    sp.coop = sp.vec_per_tok >= 2 * kWorkers ? 1 : 0;
    if (sp.stages < 2) return cudaErrorInvalidValue;   // rows too large (create() prevents it)
    sp.wait_limit_ns = 2000000000ull;
    const int smem = sp.stages * stage_bytes;
    static bool attr[kMaxDevices] = {};   // per device: attributes are per device
    const int dev = device_slot();
    if (dev < 0 || !attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(staged_rows_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemBudget);
        if (e != cudaSuccess) return e;
        if (dev >= 0) attr[dev] = true;
    }
    const int n_blocks = (sp.n_tok + sp.tok_per_block - 1) / sp.tok_per_block;
    const int grid = std::min(n_blocks, num_sms());
    staged_rows_kernel<<<grid, kThreads, smem, st>>>(sp);
    return cudaGetLastError();
}
}  // namespace

int num_sms() {
    static int n[kMaxDevices] = {};   // per device: devices may differ
    const int dev = device_slot();
    if (dev >= 0 && n[dev] > 0) return n[dev];
    int v = 0;
    if (dev < 0 || cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        v <= 0) {
        (void)cudaGetLastError();
        return 148;   // no readable device (host-only planning calls)
    }
    n[dev] = v;
    return v;
}

cudaError_t launch_kv_append(const AppendParams& p, cudaStream_t st) {
    if (p.n_tok <= 0) return cudaSuccess;
    StagedParams sp;
    sp.a_src = reinterpret_cast<const uint8_t*>(p.k_src);
    sp.b_src = reinterpret_cast<const uint8_t*>(p.v_src);
    sp.a_dst = reinterpret_cast<uint8_t*>(p.k_dst);
    sp.b_dst = reinterpret_cast<uint8_t*>(p.v_dst);
    sp.rot_a = p.rope;
    sp.rot_b = 0;
    sp.a_lo = static_cast<const uint8_t*>(p.k_lo);
    sp.a_hi = static_cast<const uint8_t*>(p.k_hi);
    sp.b_lo = static_cast<const uint8_t*>(p.v_lo);
    sp.b_hi = static_cast<const uint8_t*>(p.v_hi);
    sp.n_tok = p.n_tok;
    sp.row_bytes = p.vec_per_tok * 16;
    sp.vec_per_tok = p.vec_per_tok;
    sp.vec_per_head_log2 = p.vec_per_head_log2;
    sp.status = p.status;
    sp.ra = p.ra;
    return launch_staged(sp, st);
}

cudaError_t launch_rope_qk(const RopeParams& p, cudaStream_t st) {
    if (p.n_tok <= 0) return cudaSuccess;
    StagedParams sp;
    sp.a_src = reinterpret_cast<const uint8_t*>(p.q);
    sp.b_src = reinterpret_cast<const uint8_t*>(p.k);
    sp.a_dst = reinterpret_cast<uint8_t*>(p.q);
    sp.b_dst = reinterpret_cast<uint8_t*>(p.k);
    sp.rot_a = 1;
    sp.rot_b = 1;
    sp.a_lo = sp.a_dst;
    sp.a_hi = sp.a_dst + size_t(p.n_tok) * p.vec_per_tok * 16;
    sp.b_lo = sp.b_dst;
    sp.b_hi = sp.b_dst + size_t(p.n_tok) * p.vec_per_tok * 16;
    sp.n_tok = p.n_tok;
    sp.row_bytes = p.vec_per_tok * 16;
    sp.vec_per_tok = p.vec_per_tok;
    sp.vec_per_head_log2 = p.vec_per_head_log2;
    sp.status = p.status;
    sp.ra = p.ra;
    return launch_staged(sp, st);
}

}  // namespace frt
