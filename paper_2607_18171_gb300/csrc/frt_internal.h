// frt_internal.h — parameter blocks shared by the host library and the kernels.
#pragma once
#include <stdint.h>
#include <cuda.h>
#include <cuda_runtime.h>

namespace frt {

// Largest frames_per_chunk * d_t/2 (t-segment cos/sin entries of one chunk, passed by value).
constexpr int kMaxTEntries = 256;
// Largest number of streams in one batched attention launch.
constexpr int kMaxBatchStreams = 32;
// Largest split-KV factor (KV ranges per query group).
constexpr int kMaxSplit = 4;

// Status codes the kernels record (frt_status values).
constexpr int kStatusTimeout = 6;   // FRT_ERR_TIMEOUT
constexpr int kStatusBounds = 7;    // FRT_ERR_BOUNDS (FRT_DEBUG builds)

// Device status block (host-mapped pinned memory): the first device error wins.
struct DeviceStatus {
    int code;      // 0 = ok, else an frt_status value
    int block;     // blockIdx.x of the CTA that reported it
    int role;      // 0 producer, 1 mma issuer, 2-3 softmax groups, 4 observer, 9 item
                   // check (attention); 100+ append / RoPE kernel
    int where;     // loop iteration or barrier id
};

// RoPE tables: the t-segment cos/sin of the chunk's F frames (by value) and the
// per-stream h/w tables (device memory, fp32 from fp64 host computation).
struct RopeArgs {
    const float2* hw;   // [grid_h][d_h/2] then [grid_w][d_w/2]
    int tpf;            // tokens per frame
    int gh, gw;         // latent grid
    int dt2, dh2, dw2;  // pairs per segment
    float2 t_tab[kMaxTEntries];  // [F][d_t/2]
};

// One pair (x0, x1) packed as bf16x2 (x0 in the low half) turned by (c, s).
// Every kernel that rotates goes through this routine, so the fused and the
// separate paths give bit-identical bf16 results.
__device__ __forceinline__ uint32_t rope_pair(uint32_t x, float c, float s) {
    const float x0 = __uint_as_float(x << 16);
    const float x1 = __uint_as_float(x & 0xFFFF0000u);
    const float y0 = __fmaf_rn(x0, c, __fmul_rn(-x1, s));
    const float y1 = __fmaf_rn(x0, s, __fmul_rn(x1, c));
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(y1), "f"(y0));
    return r;
}

// t_tab: the chunk's t-segment table, either a.t_tab itself (parameter space) or a
// shared-memory copy of it (kernels whose lanes index it divergently). The h/w table is
// read-only for the whole launch, so it is read through the non-coherent path: those
// loads may then be issued ahead of the caller's stores of rotated values instead of
// waiting behind each one.
__device__ __forceinline__ float2 rope_cs(const RopeArgs& a, const float2* t_tab, int pi, int f,
                                          int r, int col) {
    if (pi < a.dt2) return t_tab[f * a.dt2 + pi];
    pi -= a.dt2;
    if (pi < a.dh2) return __ldg(&a.hw[r * a.dh2 + pi]);
    pi -= a.dh2;
    return __ldg(&a.hw[a.gh * a.dh2 + col * a.dw2 + pi]);
}

// Rotate 8 consecutive head_dim elements [d0, d0+8) (d0 % 8 == 0) of a token at
// frame f, row r, column col.
__device__ __forceinline__ uint4 rope_rotate8(uint4 v, int d0, int f, int r, int col,
                                              const RopeArgs& a, const float2* t_tab) {
    const int p0 = d0 >> 1;
    float2 cs;
    cs = rope_cs(a, t_tab, p0 + 0, f, r, col); v.x = rope_pair(v.x, cs.x, cs.y);
    cs = rope_cs(a, t_tab, p0 + 1, f, r, col); v.y = rope_pair(v.y, cs.x, cs.y);
    cs = rope_cs(a, t_tab, p0 + 2, f, r, col); v.z = rope_pair(v.z, cs.x, cs.y);
    cs = rope_cs(a, t_tab, p0 + 3, f, r, col); v.w = rope_pair(v.w, cs.x, cs.y);
    return v;
}

// ----------------------------------------------------------------------------------------
// Attention launch parameters
// ----------------------------------------------------------------------------------------
struct AttnStreamDesc {
    CUtensorMap q_map;   // 3D (D, H, Nq), box (64, 1, 128), 128-byte swizzle
    CUtensorMap k_map;   // 3D (D, H, Nkv), box (64, 1, 128)
    CUtensorMap v_map;
    CUtensorMap out_map; // 3D (D, H, Nq) over out: fp32 box (32, 1, 128) or bf16 box (64, 1, 128)
    void* out;           // [Nq, H, D] fp32 or bf16
    int n_q;
    int n_kv;
    int n_qpairs;        // ceil(Nq / 256): query groups per head
    int group_begin;     // first query group (head, 256 rows) of this stream, launch order
};

template <int MAXS>
struct AttnParams {
    AttnStreamDesc s[MAXS];
    int n_streams;
    int heads;
    int total_items;
    int out_bf16;
    float scale_log2;            // sm_scale * log2(e)
    // Split-KV of the tail: query groups [0, n_full) run whole, one item each; each later
    // group (tail group t = group - n_full) has its KV tiles cut into n_split contiguous
    // ranges processed by separate CTAs; each writes an unnormalised partial (O, running
    // max, row sum) and the last to finish merges them. n_full == groups uses none of these.
    int n_full;
    int n_split;
    CUtensorMap part_map;        // 2D (D, tail groups * n_split * 256) fp32 over part_o, box (32, 128)
    float* part_o;               // [tail groups * n_split][2][128][D] fp32
    float2* part_ml;             // [tail groups * n_split][2][128] (max in log2 units, sum)
    int* counters;               // [tail groups], zero between launches
    unsigned long long wait_limit_ns;
    DeviceStatus* status;
    // extents the FRT_DEBUG build checks every work item's indices against
    int groups_total;            // query groups of the launch
    long long part_rows_cap;     // partial rows the scratch holds
    long long tails_cap;         // merge counters the scratch holds
    RopeArgs rope;               // RoPE-Q prologue (single-stream fused path only)
};

struct AppendParams {
    const uint4* k_src;     // [Nq, H, D] bf16
    const uint4* v_src;
    uint4* k_dst;           // cache rows of the slot
    uint4* v_dst;
    int n_tok;
    int vec_per_tok;        // H * D / 8
    int vec_per_head_log2;  // log2(D / 8)
    int rope;               // rotate K on the way
    DeviceStatus* status;   // bounded-wait timeouts are recorded here
    const void* k_lo;       // the ring buffers' extents [lo, hi): the FRT_DEBUG build checks
    const void* k_hi;       // every store against them
    const void* v_lo;
    const void* v_hi;
    RopeArgs ra;
};

struct RopeParams {
    uint4* q;
    uint4* k;
    int n_tok;
    int vec_per_tok;
    int vec_per_head_log2;
    DeviceStatus* status;
    RopeArgs ra;
};

// ----------------------------------------------------------------------------------------
// Linear projections (C = A . B^T, bf16 operands, fp32 accumulation)
// ----------------------------------------------------------------------------------------
constexpr int kEpiPlain = 0;   // C row-major, fp32 or bf16
constexpr int kEpiQkv = 1;     // DiT-block QKV projection: q -> q_out, k/v -> cache slot

struct GemmParams {
    CUtensorMap a_map;      // 3D (64, M, K / 64) bf16, box (64, 128, 2) when kview3, else
                            // 2D (K, M), box (64, 128); 128-byte swizzle
    CUtensorMap b_map;      // the same over B [N, K], box rows BN / CTAs per tile
    CUtensorMap out_map[3]; // TMA store maps, 128-byte swizzle, box (128 bytes of columns,
                            // 128 rows): plain [0] over C (N, M); QKV [0..2] over q, k, v (d, M)
    int kview3;             // both maps are 3D k-block views (K a multiple of 64)
    int M, N, K;
    int tiles_m, tiles_n;   // filled in by launch_gemm
    int epi;
    // plain epilogue
    void* c;
    int ldc;                // elements
    int c_bf16;
    // QKV epilogue: N = 3 d, d = heads * head_dim, each destination [M, d] bf16
    int d;
    int head_dim;
    uint16_t* q_out;
    uint16_t* k_out;
    uint16_t* v_out;
    int rope;               // rotate q and k (3D RoPE at the chunk's positions)
    unsigned long long wait_limit_ns;
    DeviceStatus* status;
    RopeArgs ra;
};

// Work split of one attention launch: query groups [0, n_full) (launch order) run whole,
// each later group is cut into n_split KV parts whose partials are merged.
struct SplitPlan {
    int n_full = 0;
    int n_split = 1;
};
// Plans a launch over `groups` query groups with tiles[g] KV tiles each (single[g] != 0:
// one 128-row query tile) on `sms` SMs: the tail split whose simulated list schedule ends
// first. At most max_split parts, every part at least two KV tiles; max_rows / max_tails
// bound the split-KV scratch (partial rows, merge counters; negative: unbounded).
SplitPlan plan_attention(const int* tiles, const unsigned char* single, int groups, int sms,
                         int max_split, long long max_rows, long long max_tails);

// Record `code` in the status block unless an earlier error is there (first one wins).
__device__ __forceinline__ void record_status(DeviceStatus* st, int code, int role, int where) {
    if (st == nullptr) return;
    volatile DeviceStatus* s = st;
    if (s->code == 0) {
        s->block = blockIdx.x;
        s->role = role;
        s->where = where;
        __threadfence_system();
        s->code = code;
    }
}

// Kernel launchers (defined in the .cu files).
cudaError_t launch_gemm(GemmParams p, cudaStream_t st);
// Column tile width the GEMM uses for this problem, and the number of CTAs per cluster
// working on each tile (the B tensor map's box height is gemm_block_n_for / gemm_cluster_m).
int gemm_block_n_for(int M, int N, int epi, int d);
int gemm_cluster_m(int M);
cudaError_t launch_rope_qk(const RopeParams& p, cudaStream_t st);
cudaError_t launch_kv_append(const AppendParams& p, cudaStream_t st);
cudaError_t launch_attention_single(const AttnParams<1>& p, int head_dim, bool rope_q,
                                    cudaStream_t st);
cudaError_t launch_attention_batched(const AttnParams<kMaxBatchStreams>& p, int head_dim,
                                     cudaStream_t st);
// SM count of the calling thread's current device (cached per device).
int num_sms();
// One-time launch set-up (function attributes, SM counts) is per device: a function
// attribute set with cudaFuncSetAttribute applies to the current device only. Launchers
// keep such state in arrays indexed by this slot: the current device's ordinal, or -1
// when it cannot be read or is beyond kMaxDevices (the set-up is then redone every call).
constexpr int kMaxDevices = 64;
inline int device_slot() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        (void)cudaGetLastError();
        return -1;
    }
    return dev;
}
// Set the thread-local message that frt_last_error() returns.
void set_last_error(const char* msg);
// Report a CUDA runtime call of the library that failed: the message is kept for
// frt_last_error() and the runtime's (non-sticky) last error is cleared, so that it does
// not surface again from the caller's next, unrelated CUDA call.
inline void clear_cuda_error() { (void)cudaGetLastError(); }

}  // namespace frt
