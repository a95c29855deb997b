// frt_rope_append.cu — the two HBM-bound kernels of the path:
//   * 3D RoPE of q and k in place (frt_rope3d_qk),
//   * KV append into the sliding-window ring slot, optionally rotating K on the way
//     (frt_kv_append_evict / the fused frt_chunk_step).
// Both stream 16-byte vectors: one warp walks the H*D/8 vectors of one token, so the
// token's (frame, row, column) is computed once per warp and every load/store is a
// fully coalesced 512-byte warp access. Loads of a lane are all issued before its
// stores (up to kUnroll vectors per tensor in flight).
#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {

namespace {
constexpr int kThreads = 256;
constexpr int kUnroll = 8;

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__global__ void __launch_bounds__(kThreads) kv_append_kernel(const __grid_constant__ AppendParams p) {
    const int lane = threadIdx.x & 31;
    const int warps_total = gridDim.x * (kThreads / 32);
    const int vpt = p.vec_per_tok;
    for (int tok = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); tok < p.n_tok;
         tok += warps_total) {
        const int f = tok / p.ra.tpf;
        const int rem = tok - f * p.ra.tpf;
        const int r = rem / p.ra.gw;
        const int col = rem - r * p.ra.gw;
        const size_t base = size_t(tok) * vpt;
        for (int v0 = lane; v0 < vpt; v0 += 32 * kUnroll) {
            uint4 kk[kUnroll], vv[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + 32 * u;
                if (v < vpt) {
                    kk[u] = ld_stream(p.k_src + base + v);
                    vv[u] = ld_stream(p.v_src + base + v);
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + 32 * u;
                if (v < vpt) {
                    uint4 k = kk[u];
                    if (p.rope) {
                        const int d0 = (v & ((1 << p.vec_per_head_log2) - 1)) * 8;
                        k = rope_rotate8(k, d0, f, r, col, p.ra);
                    }
                    p.k_dst[base + v] = k;
                    p.v_dst[base + v] = vv[u];
                }
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads) rope_qk_kernel(const __grid_constant__ RopeParams p) {
    const int lane = threadIdx.x & 31;
    const int warps_total = gridDim.x * (kThreads / 32);
    const int vpt = p.vec_per_tok;
    for (int tok = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); tok < p.n_tok;
         tok += warps_total) {
        const int f = tok / p.ra.tpf;
        const int rem = tok - f * p.ra.tpf;
        const int r = rem / p.ra.gw;
        const int col = rem - r * p.ra.gw;
        const size_t base = size_t(tok) * vpt;
        for (int v0 = lane; v0 < vpt; v0 += 32 * kUnroll) {
            uint4 qq[kUnroll], kk[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + 32 * u;
                if (v < vpt) {
                    qq[u] = p.q[base + v];
                    kk[u] = p.k[base + v];
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + 32 * u;
                if (v < vpt) {
                    const int d0 = (v & ((1 << p.vec_per_head_log2) - 1)) * 8;
                    p.q[base + v] = rope_rotate8(qq[u], d0, f, r, col, p.ra);
                    p.k[base + v] = rope_rotate8(kk[u], d0, f, r, col, p.ra);
                }
            }
        }
    }
}

int grid_for_tokens(int n_tok) {
    // enough resident warps to keep ~64 KB per SM in flight; never more CTAs than tokens need
    const int per_cta = kThreads / 32;
    int want = num_sms() * 8;
    int need = (n_tok + per_cta - 1) / per_cta;
    return want < need ? want : (need > 0 ? need : 1);
}
}  // namespace

int num_sms() {
    static int n = 0;
    if (n == 0) {
        int dev = 0, v = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
            n = v;
        else
            n = 148;
    }
    return n;
}

cudaError_t launch_kv_append(const AppendParams& p, cudaStream_t st) {
    if (p.n_tok <= 0) return cudaSuccess;
    kv_append_kernel<<<grid_for_tokens(p.n_tok), kThreads, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_rope_qk(const RopeParams& p, cudaStream_t st) {
    if (p.n_tok <= 0) return cudaSuccess;
    rope_qk_kernel<<<grid_for_tokens(p.n_tok), kThreads, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace frt
