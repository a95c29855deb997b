// frt_host.cu — the C ABI (include/frt.h): per-stream persistent state (the rolling KV
// cache), host-side window arithmetic, argument/state checks, TMA descriptor encoding and
// kernel launches on the caller's CUDA stream.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/frt.h"
#include "frt_internal.h"

using namespace frt;

namespace {

thread_local std::string g_last_error;

frt_status fail(frt_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

frt_status cuda_fail(cudaError_t e, const char* what) {
    clear_cuda_error();
    return fail(e == cudaErrorMemoryAllocation ? FRT_ERR_OOM : FRT_ERR_CUDA, "%s: %s", what,
                cudaGetErrorString(e));
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 3D map over a token-major [rows, heads, head_dim] bf16 tensor; box = 64 dims x 1 head x
// 128 rows, 128-byte swizzle; rows past `rows` read as zero.
frt_status make_map(CUtensorMap* map, const void* base, int head_dim, int heads, long long rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[3] = {cuuint64_t(head_dim), cuuint64_t(heads), cuuint64_t(rows)};
    cuuint64_t strides[2] = {cuuint64_t(head_dim) * 2, cuuint64_t(heads) * head_dim * 2};
    cuuint32_t box[3] = {64, 1, 128};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
    return FRT_OK;
}

// 3D map over an attention output [rows, heads, head_dim] (fp32 or bf16) for TMA stores:
// box = 128 bytes of head_dim x 1 head x 128 rows, 128-byte swizzle; rows past `rows` are
// not written.
frt_status make_out_map(CUtensorMap* map, void* base, int head_dim, int heads, long long rows,
                        bool bf16) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    const int es = bf16 ? 2 : 4;
    cuuint64_t dims[3] = {cuuint64_t(head_dim), cuuint64_t(heads), cuuint64_t(rows)};
    cuuint64_t strides[2] = {cuuint64_t(head_dim) * es, cuuint64_t(heads) * head_dim * es};
    cuuint32_t box[3] = {cuuint32_t(128 / es), 1, 128};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
                    3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
    return FRT_OK;
}

// 2D fp32 map over split-KV partial rows [rows, head_dim]: box 32 columns x 128 rows,
// 128-byte swizzle (the layout the attention kernel stages its partial tiles in).
frt_status make_part_map(CUtensorMap* map, float* base, int head_dim, long long rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    if (rows >= (1LL << 31)) return fail(FRT_ERR_UNSUPPORTED, "split-KV scratch too large");
    cuuint64_t dims[2] = {cuuint64_t(head_dim), cuuint64_t(rows)};
    cuuint64_t strides[1] = {cuuint64_t(head_dim) * 4};
    cuuint32_t box[2] = {32, 128};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
    return FRT_OK;
}

// 2D store map over a row-major [rows, cols] fp32 or bf16 matrix with a leading dimension
// of ld elements; box = 128 bytes of columns x 128 rows, 128-byte swizzle (the layout the
// projection kernel stages its output units in); past the extent nothing is written.
frt_status make_store_map_2d(CUtensorMap* map, void* base, long long cols, long long rows,
                             long long ld, bool bf16) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    const int es = bf16 ? 2 : 4;
    cuuint64_t dims[2] = {cuuint64_t(cols), cuuint64_t(rows)};
    cuuint64_t strides[1] = {cuuint64_t(ld) * es};
    cuuint32_t box[2] = {cuuint32_t(128 / es), 128};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
                    2, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
    return FRT_OK;
}

// 2D map over a row-major [rows, K] bf16 matrix; box = 64 columns x box_rows rows,
// 128-byte swizzle; rows and columns past the extent read as zero.
frt_status make_map_2d(CUtensorMap* map, const void* base, long long K, long long rows,
                       int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[2] = {cuuint64_t(K), cuuint64_t(rows)};
    cuuint64_t strides[1] = {cuuint64_t(K) * 2};
    cuuint32_t box[2] = {64, cuuint32_t(box_rows)};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(FRT_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
    return FRT_OK;
}

// 3D view (64, rows, K / 64) of a row-major [rows, K] bf16 matrix (K a multiple of 64):
// element (c, r, kb) is column 64 kb + c of row r, so one box (64, box_rows, 2) carries two
// consecutive 64-column k-blocks of box_rows rows, laid out k-block after k-block.
CUresult encode_kview(CUtensorMap* map, const void* base, long long K, long long rows,
                      int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return CUDA_ERROR_NOT_SUPPORTED;
    cuuint64_t dims[3] = {64, cuuint64_t(rows), cuuint64_t(K / 64)};
    cuuint64_t strides[2] = {cuuint64_t(K) * 2, 128};
    cuuint32_t box[3] = {64, cuuint32_t(box_rows), 2};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Operand maps of C = A B^T (A [M, K], B [N, K] row-major bf16): k-block views when K is
// a multiple of 64 and the driver takes them, else 2D maps (the kernel then issues one
// copy per k-block).
frt_status make_gemm_maps(GemmParams& g, const void* a, const void* b, long long K, long long M,
                          long long N, int b_box_rows) {
    if (K % 64 == 0 && encode_kview(&g.a_map, a, K, M, 128) == CUDA_SUCCESS &&
        encode_kview(&g.b_map, b, K, N, b_box_rows) == CUDA_SUCCESS) {
        g.kview3 = 1;
        return FRT_OK;
    }
    g.kview3 = 0;
    frt_status st = make_map_2d(&g.a_map, a, K, M, 128);
    return st != FRT_OK ? st : make_map_2d(&g.b_map, b, K, N, b_box_rows);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

enum Phase { kStart = 0, kRoped = 1, kAppended = 2 };

constexpr unsigned long long kDefaultWaitLimitNs = 2000000000ull;  // 2 s per bounded wait

// Guard words: kGuardBytes of kGuardByte before and after each cache buffer (one
// allocation each), written at configure and compared by frt_stream_check_guards. A
// kernel that wrote past either end of the ring would change them.
constexpr size_t kGuardBytes = 256;
constexpr unsigned char kGuardByte = 0xA7;
#ifdef FRT_DEBUG
constexpr bool kDebugBuild = true;
// the debug build also keeps one chunk of slack after the rear guard (filled like the
// guard): a write one slot past the ring that a bounds check missed would still land in
// the library's own memory, and the guard check would report it
constexpr bool kSlackChunk = true;
// self-test hook: the next append targets ring slot W (one past the ring)
int g_append_past_ring = 0;
#else
constexpr bool kDebugBuild = false;
constexpr bool kSlackChunk = false;
#endif

// staging sets of the host-buffer step (frt_chunk_step_host)
constexpr int kStageSets = 3;

}  // namespace

struct frt_stream {
    int heads, head_dim, tpf, frames, window, n_q;
    bool configured = false;
    frt_config cfg{};
    float scale = 0.f;
    cudaStream_t cs = nullptr;
    void* cache_k = nullptr;    // ring buffers, kGuardBytes into their allocations
    void* cache_v = nullptr;
    unsigned char* alloc_k = nullptr;   // the allocations (guard, ring, guard [, slack])
    unsigned char* alloc_v = nullptr;
    size_t rear_bytes = 0;              // guard (+ slack) after each ring
    size_t chunk_elems = 0;     // Nq * H * D
    float2* d_hw = nullptr;     // h/w RoPE tables
    int hw_entries = 0;
    DeviceStatus* status_host = nullptr;
    DeviceStatus* status_dev = nullptr;
    long long counter = 0;
    int phase = kStart;
    const void* last_q = nullptr;
    const void* last_k = nullptr;
    const void* last_v = nullptr;
    void* stage = nullptr;      // host-API staging: two sets of q, k, v (bf16) and out
    size_t stage_bytes = 0;
    int stage_turn = 0;         // staging set of the next host-buffer step (of kStageSets)
    cudaStream_t cp_in = nullptr;   // host-to-device copies of host-buffer steps
    cudaStream_t cp_out = nullptr;  // device-to-host copies of host-buffer steps
    cudaEvent_t ev_in[kStageSets] = {};    // inputs of set b landed
    cudaEvent_t ev_done[kStageSets] = {};  // kernels reading set b finished
    cudaEvent_t ev_out[kStageSets] = {};   // output of set b copied out
    unsigned long long wait_limit_ns = kDefaultWaitLimitNs;
    cudaEvent_t ev = nullptr;   // cross-stream ordering for batched launches
    cudaEvent_t attn_start = nullptr;  // caller-owned instrumentation events
    cudaEvent_t attn_stop = nullptr;
    cudaEvent_t app_start = nullptr;
    cudaEvent_t app_stop = nullptr;
    cudaEvent_t qkv_start = nullptr;   // frt_block_step projections
    cudaEvent_t qkv_stop = nullptr;
    cudaEvent_t proj_start = nullptr;
    cudaEvent_t proj_stop = nullptr;
    // split-KV scratch: partial O / (max, sum) rows per (tail group, split), one counter
    // per tail group (zero between launches)
    float* part_o = nullptr;
    float2* part_ml = nullptr;
    int* counters = nullptr;
    long long part_rows = 0;     // capacity: partial rows (256 per tail group and split)
    long long part_tails = 0;    // capacity: tail groups (merge counters)
    // work split of this stream's attention launch for each window fill n_valid = 1..W
    // (index n_valid - 1), planned once at configure
    std::vector<SplitPlan> plans;
};

namespace {

frt_status check_device_status(frt_stream_t* s) {
    if (s->status_host == nullptr) return FRT_OK;
    volatile DeviceStatus* st = s->status_host;
    int code = st->code;
    if (code == FRT_ERR_BOUNDS)
        return fail(FRT_ERR_BOUNDS,
                    "device bounds check failed (block %d, role %d, at %d); reset the stream",
                    st->block, st->role, st->where);
    if (code != 0)
        return fail(static_cast<frt_status>(code),
                    "device wait gave up (block %d, role %d, at %d); reset the stream", st->block,
                    st->role, st->where);
    return FRT_OK;
}

frt_status require_configured(frt_stream_t* s) {
    if (s == nullptr) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if (!s->configured) return fail(FRT_ERR_STATE, "stream not configured");
    return check_device_status(s);
}

// RoPE argument block for chunk `c` (t-segment cos/sin of its frames, fp64 -> fp32).
void fill_rope(const frt_stream_t* s, long long c, RopeArgs& a) {
    a.hw = s->d_hw;
    a.tpf = s->tpf;
    a.gh = s->cfg.grid_h;
    a.gw = s->cfg.grid_w;
    a.dt2 = s->cfg.rope_dt / 2;
    a.dh2 = s->cfg.rope_dh / 2;
    a.dw2 = s->cfg.rope_dw / 2;
    const double theta = s->cfg.theta;
    for (int f = 0; f < s->frames; ++f) {
        const double t = double(c) * s->frames + f;
        for (int j = 0; j < a.dt2; ++j) {
            const double ang = t * std::pow(theta, -2.0 * j / double(s->cfg.rope_dt));
            a.t_tab[f * a.dt2 + j] = make_float2(float(std::cos(ang)), float(std::sin(ang)));
        }
    }
}

// Make sure s owns split-KV scratch for `rows` partial rows and `tails` merge counters
// (allocates, synchronously, only when it must grow).
frt_status ensure_scratch(frt_stream_t* s, long long rows, long long tails) {
    if (rows <= s->part_rows && tails <= s->part_tails) return FRT_OK;
    cudaError_t e;
    if (s->part_o && (e = cudaStreamSynchronize(s->cs)) != cudaSuccess)
        return cuda_fail(e, "sync before scratch growth");
    const long long r = std::max(rows, s->part_rows);
    const long long t = std::max(std::max(tails, s->part_tails), 1LL);
    if (s->part_o) cudaFree(s->part_o);
    if (s->part_ml) cudaFree(s->part_ml);
    if (s->counters) cudaFree(s->counters);
    s->part_o = nullptr;
    s->part_ml = nullptr;
    s->counters = nullptr;
    s->part_rows = 0;
    s->part_tails = 0;
    if ((e = cudaMalloc(&s->part_o, size_t(std::max(r, 256LL)) * s->head_dim * sizeof(float))) !=
            cudaSuccess ||
        (e = cudaMalloc(&s->part_ml, size_t(std::max(r, 256LL)) * sizeof(float2))) != cudaSuccess ||
        (e = cudaMalloc(&s->counters, size_t(t) * sizeof(int))) != cudaSuccess ||
        (e = cudaMemset(s->counters, 0, size_t(t) * sizeof(int))) != cudaSuccess ||
        (e = cudaDeviceSynchronize()) != cudaSuccess)
        return cuda_fail(e, "split-KV scratch allocation");
    s->part_rows = std::max(r, 256LL);
    s->part_tails = t;
    return FRT_OK;
}

// Query groups of one stream in launch order (head-major): KV tiles and whether the
// group has a single 128-row query tile (the ragged last group of each head).
void stream_groups(int n_q, int heads, long long n_kv, std::vector<int>& tiles,
                   std::vector<unsigned char>& single) {
    const int pairs = (n_q + 255) / 256;
    const int t = int((n_kv + 127) / 128);
    for (int h = 0; h < heads; ++h)
        for (int pr = 0; pr < pairs; ++pr) {
            tiles.push_back(t);
            single.push_back((pr * 256 + 128) >= n_q ? 1 : 0);
        }
}

// Split-KV scratch of a launch: partial rows and merge counters.
long long plan_rows(const SplitPlan& pl, long long groups) {
    return pl.n_split > 1 ? (groups - pl.n_full) * pl.n_split * 256 : 0;
}
long long plan_tails(const SplitPlan& pl, long long groups) {
    return pl.n_split > 1 ? groups - pl.n_full : 0;
}

int log2_exact(int x) {
    int l = 0;
    while ((1 << l) < x) ++l;
    return l;
}

// out_bf16: 1 / 0 force the output dtype, -1 takes the stream's configured one.
frt_status attention_single(frt_stream_t* s, const void* q, void* out, bool rope_q,
                            int out_bf16 = -1) {
    AttnParams<1> p;
    std::memset(&p, 0, sizeof(p));
    const long long n_valid = std::min<long long>(s->counter, s->window);
    AttnStreamDesc& d = p.s[0];
    frt_status st;
    if ((st = make_map(&d.q_map, q, s->head_dim, s->heads, s->n_q)) != FRT_OK) return st;
    const long long n_kv = n_valid * s->n_q;
    if ((st = make_map(&d.k_map, s->cache_k, s->head_dim, s->heads, n_kv)) != FRT_OK) return st;
    if ((st = make_map(&d.v_map, s->cache_v, s->head_dim, s->heads, n_kv)) != FRT_OK) return st;
    d.out = out;
    d.n_q = s->n_q;
    d.n_kv = int(n_kv);
    d.n_qpairs = (s->n_q + 255) / 256;
    d.group_begin = 0;
    const long long groups = (long long)d.n_qpairs * s->heads;
    const SplitPlan pl = s->plans[size_t(n_valid - 1)];
    if (plan_rows(pl, groups) > s->part_rows || plan_tails(pl, groups) > s->part_tails)
        return fail(FRT_ERR_STATE, "split-KV scratch smaller than the configured plan");
    p.n_full = pl.n_full;
    p.n_split = pl.n_split;
    p.part_o = s->part_o;
    p.part_ml = s->part_ml;
    p.counters = s->counters;
    p.groups_total = int(groups);
    p.part_rows_cap = s->part_rows;
    p.tails_cap = s->part_tails;
    p.n_streams = 1;
    p.heads = s->heads;
    p.total_items = int(pl.n_full + (groups - pl.n_full) * pl.n_split);
    p.out_bf16 = out_bf16 >= 0 ? out_bf16 : (s->cfg.out_dtype == FRT_OUT_BF16);
    if ((st = make_out_map(&d.out_map, out, s->head_dim, s->heads, s->n_q, p.out_bf16 != 0)) !=
        FRT_OK)
        return st;
    if (p.n_split > 1 &&
        (st = make_part_map(&p.part_map, s->part_o, s->head_dim, s->part_rows)) != FRT_OK)
        return st;
    p.scale_log2 = float(double(s->scale) * 1.4426950408889634);
    p.wait_limit_ns = s->wait_limit_ns;
    p.status = s->status_dev;
    if (rope_q) fill_rope(s, s->counter - 1, p.rope);
    cudaError_t e = cudaSuccess;
    if (s->attn_start) e = cudaEventRecord(s->attn_start, s->cs);
    if (e == cudaSuccess) e = launch_attention_single(p, s->head_dim, rope_q, s->cs);
    if (e == cudaSuccess && s->attn_stop) e = cudaEventRecord(s->attn_stop, s->cs);
    if (e != cudaSuccess) return cuda_fail(e, "attention launch");
    return FRT_OK;
}

frt_status append_impl(frt_stream_t* s, const void* k, const void* v, bool rope_k, int* slot_out,
                       long long* evicted_out) {
    int slot;
    long long evicted;
    frt_window_index(s->counter, s->window, &slot, &evicted, nullptr);
    AppendParams p;
    std::memset(&p, 0, sizeof(p));
    size_t off = size_t(slot) * s->chunk_elems;
#ifdef FRT_DEBUG
    if (g_append_past_ring) {   // self-test: aim one slot past the ring
        off = size_t(s->window) * s->chunk_elems;
        g_append_past_ring = 0;
    }
#endif
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    p.k_lo = s->cache_k;
    p.k_hi = static_cast<const uint8_t*>(s->cache_k) + cache_bytes;
    p.v_lo = s->cache_v;
    p.v_hi = static_cast<const uint8_t*>(s->cache_v) + cache_bytes;
    p.k_src = static_cast<const uint4*>(k);
    p.v_src = static_cast<const uint4*>(v);
    p.k_dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(s->cache_k) + off);
    p.v_dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(s->cache_v) + off);
    p.n_tok = s->n_q;
    p.vec_per_tok = s->heads * s->head_dim / 8;
    p.vec_per_head_log2 = log2_exact(s->head_dim / 8);
    p.rope = rope_k ? 1 : 0;
    p.status = s->status_dev;
    if (rope_k) fill_rope(s, s->counter, p.ra);
    cudaError_t e = cudaSuccess;
    if (s->app_start) e = cudaEventRecord(s->app_start, s->cs);
    if (e == cudaSuccess) e = launch_kv_append(p, s->cs);
    if (e == cudaSuccess && s->app_stop) e = cudaEventRecord(s->app_stop, s->cs);
    if (e != cudaSuccess) return cuda_fail(e, "append launch");
    s->counter += 1;
    s->phase = kAppended;
    s->last_k = k;
    s->last_v = v;
    if (slot_out) *slot_out = slot;
    if (evicted_out) *evicted_out = evicted;
    return FRT_OK;
}

void free_device(frt_stream_t* s) {
    if (s->alloc_k) cudaFree(s->alloc_k);
    if (s->alloc_v) cudaFree(s->alloc_v);
    s->alloc_k = s->alloc_v = nullptr;
    if (s->d_hw) cudaFree(s->d_hw);
    if (s->stage) cudaFree(s->stage);
    if (s->status_host) cudaFreeHost(s->status_host);
    if (s->ev) cudaEventDestroy(s->ev);
    s->ev = nullptr;
    if (s->cp_in) cudaStreamSynchronize(s->cp_in);
    if (s->cp_out) cudaStreamSynchronize(s->cp_out);
    for (int b = 0; b < kStageSets; ++b) {
        if (s->ev_in[b]) cudaEventDestroy(s->ev_in[b]);
        if (s->ev_done[b]) cudaEventDestroy(s->ev_done[b]);
        if (s->ev_out[b]) cudaEventDestroy(s->ev_out[b]);
        s->ev_in[b] = s->ev_done[b] = s->ev_out[b] = nullptr;
    }
    if (s->cp_in) cudaStreamDestroy(s->cp_in);
    if (s->cp_out) cudaStreamDestroy(s->cp_out);
    s->cp_in = s->cp_out = nullptr;
    if (s->part_o) cudaFree(s->part_o);
    if (s->part_ml) cudaFree(s->part_ml);
    if (s->counters) cudaFree(s->counters);
    s->part_o = nullptr;
    s->part_ml = nullptr;
    s->counters = nullptr;
    s->part_rows = 0;
    s->part_tails = 0;
    s->cache_k = s->cache_v = nullptr;
    s->d_hw = nullptr;
    s->stage = nullptr;
    s->status_host = s->status_dev = nullptr;
}

}  // namespace

extern "C" {

const char* frt_version(void) { return "frt 0.1 (sm_103a)"; }

const char* frt_last_error(void) { return g_last_error.c_str(); }

const char* frt_status_string(frt_status st) {
    switch (st) {
        case FRT_OK: return "FRT_OK";
        case FRT_ERR_INVALID_ARG: return "FRT_ERR_INVALID_ARG";
        case FRT_ERR_STATE: return "FRT_ERR_STATE";
        case FRT_ERR_OOM: return "FRT_ERR_OOM";
        case FRT_ERR_CUDA: return "FRT_ERR_CUDA";
        case FRT_ERR_UNSUPPORTED: return "FRT_ERR_UNSUPPORTED";
        case FRT_ERR_TIMEOUT: return "FRT_ERR_TIMEOUT";
        case FRT_ERR_BOUNDS: return "FRT_ERR_BOUNDS";
    }
    return "FRT_ERR_UNKNOWN";
}

frt_status frt_window_index(long long chunk, int window, int* slot, long long* evicted,
                            int* valid_chunks) {
    if (chunk < 0 || window < 1) return fail(FRT_ERR_INVALID_ARG, "chunk >= 0 and window >= 1");
    if (slot) *slot = int(chunk % window);
    if (evicted) *evicted = chunk >= window ? chunk - window : -1;
    if (valid_chunks) *valid_chunks = int(chunk + 1 < window ? chunk + 1 : window);
    return FRT_OK;
}

frt_stream_t* frt_stream_create(int heads, int head_dim, int tokens_per_frame,
                                int frames_per_chunk, int window_chunks) {
    if (heads < 1 || tokens_per_frame < 1 || frames_per_chunk < 1 || window_chunks < 1) {
        fail(FRT_ERR_INVALID_ARG, "heads, tokens_per_frame, frames_per_chunk, window >= 1");
        return nullptr;
    }
    if (head_dim != 64 && head_dim != 128) {
        fail(FRT_ERR_UNSUPPORTED, "head_dim %d unsupported (64 or 128)", head_dim);
        return nullptr;
    }
    const long long n_q = (long long)frames_per_chunk * tokens_per_frame;
    if ((long long)heads * head_dim > 12800) {
        // the staged append/RoPE kernel keeps 4 stages of two token rows in 200 KB of
        // shared memory: a token row (heads * head_dim bf16) may be at most 25 KB
        fail(FRT_ERR_UNSUPPORTED, "heads * head_dim = %lld exceeds 12800",
             (long long)heads * head_dim);
        return nullptr;
    }
    if (n_q > (1 << 20) || n_q * window_chunks > (1 << 24)) {
        fail(FRT_ERR_UNSUPPORTED, "chunk or window too large (Nq=%lld, W=%d)", n_q, window_chunks);
        return nullptr;
    }
    frt_stream_t* s = new (std::nothrow) frt_stream();
    if (!s) {
        fail(FRT_ERR_OOM, "host allocation failed");
        return nullptr;
    }
    s->heads = heads;
    s->head_dim = head_dim;
    s->tpf = tokens_per_frame;
    s->frames = frames_per_chunk;
    s->window = window_chunks;
    s->n_q = int(n_q);
    s->chunk_elems = size_t(n_q) * heads * head_dim;
    frt_config_default(s, &s->cfg);
    return s;
}

frt_status frt_config_default(const frt_stream_t* s, frt_config* cfg) {
    if (!s || !cfg) return fail(FRT_ERR_INVALID_ARG, "NULL argument");
    const int D = s->head_dim;
    int dt = 2 * int(std::lround(D / 8.0));
    int dh = 2 * ((D - dt) / 4);
    cfg->grid_h = 1;
    cfg->grid_w = s->tpf;
    cfg->rope_dt = dt;
    cfg->rope_dh = dh;
    cfg->rope_dw = D - dt - dh;
    cfg->theta = 10000.0;
    cfg->sm_scale = 1.0 / std::sqrt(double(D));
    cfg->out_dtype = FRT_OUT_F32;
    cfg->cuda_stream = nullptr;
    return FRT_OK;
}

frt_status frt_stream_configure(frt_stream_t* s, const frt_config* cfg) {
    if (!s || !cfg) return fail(FRT_ERR_INVALID_ARG, "NULL argument");
    if (cfg->grid_h < 1 || cfg->grid_w < 1 || (long long)cfg->grid_h * cfg->grid_w != s->tpf)
        return fail(FRT_ERR_INVALID_ARG, "grid_h * grid_w must equal tokens_per_frame");
    if (cfg->rope_dt < 0 || cfg->rope_dh < 0 || cfg->rope_dw < 0 || (cfg->rope_dt & 1) ||
        (cfg->rope_dh & 1) || (cfg->rope_dw & 1) ||
        cfg->rope_dt + cfg->rope_dh + cfg->rope_dw != s->head_dim)
        return fail(FRT_ERR_INVALID_ARG, "rope split must be even and sum to head_dim");
    if (!(cfg->theta > 1.0)) return fail(FRT_ERR_INVALID_ARG, "theta must be > 1");
    if (cfg->out_dtype != FRT_OUT_F32 && cfg->out_dtype != FRT_OUT_BF16)
        return fail(FRT_ERR_INVALID_ARG, "unknown out_dtype");
    if ((long long)s->frames * (cfg->rope_dt / 2) > kMaxTEntries)
        return fail(FRT_ERR_UNSUPPORTED, "frames_per_chunk * d_t/2 exceeds %d", kMaxTEntries);
    if (s->configured) {
        cudaError_t e = cudaStreamSynchronize(s->cs);
        if (e != cudaSuccess) return cuda_fail(e, "sync before reconfigure");
    }
    // a configure that fails part-way leaves the stream unconfigured, never half-built:
    // later calls return FRT_ERR_STATE until a configure succeeds
    s->configured = false;
    s->cfg = *cfg;
    s->scale = float(cfg->sm_scale > 0 ? cfg->sm_scale : 1.0 / std::sqrt(double(s->head_dim)));
    s->cs = static_cast<cudaStream_t>(cfg->cuda_stream);

    cudaError_t e;
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    if (!s->cache_k) {
        s->rear_bytes = kGuardBytes + (kSlackChunk ? s->chunk_elems * 2 : 0);
        const size_t total = kGuardBytes + cache_bytes + s->rear_bytes;
        if ((e = cudaMalloc(reinterpret_cast<void**>(&s->alloc_k), total)) != cudaSuccess ||
            (e = cudaMalloc(reinterpret_cast<void**>(&s->alloc_v), total)) != cudaSuccess) {
            free_device(s);
            return cuda_fail(e, "cache allocation");
        }
        s->cache_k = s->alloc_k + kGuardBytes;
        s->cache_v = s->alloc_v + kGuardBytes;
        for (unsigned char* a : {s->alloc_k, s->alloc_v})
            if ((e = cudaMemset(a, kGuardByte, kGuardBytes)) != cudaSuccess ||
                (e = cudaMemset(a + kGuardBytes + cache_bytes, kGuardByte, s->rear_bytes)) !=
                    cudaSuccess) {
                free_device(s);
                return cuda_fail(e, "guard words");
            }
    }
    if (!s->status_host) {
        if ((e = cudaHostAlloc(reinterpret_cast<void**>(&s->status_host), sizeof(DeviceStatus),
                               cudaHostAllocMapped)) != cudaSuccess ||
            (e = cudaHostGetDevicePointer(reinterpret_cast<void**>(&s->status_dev),
                                          s->status_host, 0)) != cudaSuccess) {
            free_device(s);
            return cuda_fail(e, "status allocation");
        }
    }
    std::memset(s->status_host, 0, sizeof(DeviceStatus));
    if (!s->ev && (e = cudaEventCreateWithFlags(&s->ev, cudaEventDisableTiming)) != cudaSuccess) {
        free_device(s);
        return cuda_fail(e, "event creation");
    }
    // h/w tables: [grid_h][d_h/2] then [grid_w][d_w/2], cos/sin computed in fp64
    const int dh2 = cfg->rope_dh / 2, dw2 = cfg->rope_dw / 2;
    std::vector<float2> hw(size_t(cfg->grid_h) * dh2 + size_t(cfg->grid_w) * dw2 + 1);
    for (int r = 0; r < cfg->grid_h; ++r)
        for (int j = 0; j < dh2; ++j) {
            const double a = r * std::pow(cfg->theta, -2.0 * j / double(cfg->rope_dh));
            hw[size_t(r) * dh2 + j] = make_float2(float(std::cos(a)), float(std::sin(a)));
        }
    for (int c = 0; c < cfg->grid_w; ++c)
        for (int j = 0; j < dw2; ++j) {
            const double a = c * std::pow(cfg->theta, -2.0 * j / double(cfg->rope_dw));
            hw[size_t(cfg->grid_h) * dh2 + size_t(c) * dw2 + j] =
                make_float2(float(std::cos(a)), float(std::sin(a)));
        }
    if (s->d_hw) cudaFree(s->d_hw);
    s->d_hw = nullptr;
    if ((e = cudaMalloc(&s->d_hw, hw.size() * sizeof(float2))) != cudaSuccess) {
        free_device(s);
        return cuda_fail(e, "rope table allocation");
    }
    if ((e = cudaMemcpy(s->d_hw, hw.data(), hw.size() * sizeof(float2),
                        cudaMemcpyHostToDevice)) != cudaSuccess)
        return cuda_fail(e, "rope table upload");
    s->hw_entries = int(hw.size());
    {
        // the work split of every window fill, and split-KV scratch for all of them
        const long long groups = (long long)((s->n_q + 255) / 256) * s->heads;
        s->plans.clear();
        long long rows = 0, tails = 0;
        for (int nv = 1; nv <= s->window; ++nv) {
            std::vector<int> tiles;
            std::vector<unsigned char> single;
            stream_groups(s->n_q, s->heads, (long long)nv * s->n_q, tiles, single);
            const SplitPlan pl = plan_attention(tiles.data(), single.data(), int(groups),
                                                num_sms(), kMaxSplit, -1, -1);
            s->plans.push_back(pl);
            rows = std::max(rows, plan_rows(pl, groups));
            tails = std::max(tails, plan_tails(pl, groups));
        }
        frt_status st = ensure_scratch(s, rows, tails);
        if (st != FRT_OK) {
            free_device(s);
            return st;
        }
    }
    // zero cache: rows past the valid prefix are never read by value, but keep them finite;
    // zero merge counters: a launch that gave up part-way may have left some counted
    if ((e = cudaMemset(s->cache_k, 0, cache_bytes)) != cudaSuccess ||
        (e = cudaMemset(s->cache_v, 0, cache_bytes)) != cudaSuccess ||
        (s->counters &&
         (e = cudaMemset(s->counters, 0, size_t(s->part_tails) * sizeof(int))) != cudaSuccess))
        return cuda_fail(e, "cache clear");
    if ((e = cudaDeviceSynchronize()) != cudaSuccess) return cuda_fail(e, "configure sync");
    s->counter = 0;
    s->phase = kStart;
    s->last_q = s->last_k = s->last_v = nullptr;
    s->configured = true;
    return FRT_OK;
}

frt_status frt_rope3d_qk(frt_stream_t* s, void* q, void* k) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!q || !k || !aligned16(q) || !aligned16(k))
        return fail(FRT_ERR_INVALID_ARG, "q and k must be non-NULL and 16-byte aligned");
    if (s->phase == kRoped) return fail(FRT_ERR_STATE, "rope called twice for one chunk");
    RopeParams p;
    std::memset(&p, 0, sizeof(p));
    p.q = static_cast<uint4*>(q);
    p.k = static_cast<uint4*>(k);
    p.n_tok = s->n_q;
    p.vec_per_tok = s->heads * s->head_dim / 8;
    p.vec_per_head_log2 = log2_exact(s->head_dim / 8);
    p.status = s->status_dev;
    fill_rope(s, s->counter, p.ra);
    cudaError_t e = launch_rope_qk(p, s->cs);
    if (e != cudaSuccess) return cuda_fail(e, "rope launch");
    s->phase = kRoped;
    s->last_q = q;
    return FRT_OK;
}

frt_status frt_kv_append_evict(frt_stream_t* s, const void* k, const void* v, int* slot_out,
                               long long* evicted_out) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!k || !v || !aligned16(k) || !aligned16(v))
        return fail(FRT_ERR_INVALID_ARG, "k and v must be non-NULL and 16-byte aligned");
    if (s->phase != kRoped) return fail(FRT_ERR_STATE, "append must follow frt_rope3d_qk");
    return append_impl(s, k, v, false, slot_out, evicted_out);
}

frt_status frt_chunk_attention(const void* q, const void* k, const void* v, void* out,
                               frt_stream_t* s) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!q || !out || !aligned16(q) || !aligned16(out))
        return fail(FRT_ERR_INVALID_ARG, "q and out must be non-NULL and 16-byte aligned");
    if (s->phase != kAppended) return fail(FRT_ERR_STATE, "attention must follow an append");
    if ((k && k != s->last_k) || (v && v != s->last_v))
        return fail(FRT_ERR_STATE, "k/v are not the tensors of the last append");
    if (q != s->last_q) return fail(FRT_ERR_STATE, "q is not the tensor rotated for this chunk");
    return attention_single(s, q, out, false);
}

frt_status frt_chunk_step(frt_stream_t* s, const void* q, const void* k, const void* v,
                          void* out, int* slot_out, long long* evicted_out) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!q || !k || !v || !out || !aligned16(q) || !aligned16(k) || !aligned16(v) ||
        !aligned16(out))
        return fail(FRT_ERR_INVALID_ARG, "q, k, v, out must be non-NULL and 16-byte aligned");
    if (s->phase == kRoped) return fail(FRT_ERR_STATE, "a separate rope is pending");
    if ((st = append_impl(s, k, v, true, slot_out, evicted_out)) != FRT_OK) return st;
    s->last_q = q;
    return attention_single(s, q, out, true);
}

frt_status frt_block_step(frt_stream_t* s, const void* x, const void* w_qkv, const void* w_o,
                          void* q_buf, void* o_buf, void* y, int* slot_out,
                          long long* evicted_out) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!x || !w_qkv || !w_o || !q_buf || !o_buf || !y || !aligned16(x) || !aligned16(w_qkv) ||
        !aligned16(w_o) || !aligned16(q_buf) || !aligned16(o_buf) || !aligned16(y))
        return fail(FRT_ERR_INVALID_ARG,
                    "x, w_qkv, w_o, q_buf, o_buf, y must be non-NULL and 16-byte aligned");
    if (s->phase == kRoped) return fail(FRT_ERR_STATE, "a separate rope is pending");
    const int d = s->heads * s->head_dim;
    if (d % 128 != 0)
        return fail(FRT_ERR_UNSUPPORTED, "heads * head_dim must be a multiple of 128");
    int slot;
    long long evicted;
    frt_window_index(s->counter, s->window, &slot, &evicted, nullptr);
    const size_t off = size_t(slot) * s->chunk_elems;

    // 1. QKV projection; its epilogue rotates q, k and writes k, v into the ring slot
    GemmParams g;
    std::memset(&g, 0, sizeof(g));
    const int bn = gemm_block_n_for(s->n_q, 3 * d, kEpiQkv, d);
    if ((st = make_gemm_maps(g, x, w_qkv, d, s->n_q, 3LL * d, bn / gemm_cluster_m(s->n_q))) != FRT_OK)
        return st;
    g.M = s->n_q;
    g.N = 3 * d;
    g.K = d;
    g.epi = kEpiQkv;
    g.d = d;
    g.head_dim = s->head_dim;
    g.q_out = static_cast<uint16_t*>(q_buf);
    g.k_out = static_cast<uint16_t*>(s->cache_k) + off;
    g.v_out = static_cast<uint16_t*>(s->cache_v) + off;
    if ((st = make_store_map_2d(&g.out_map[0], g.q_out, d, s->n_q, d, true)) != FRT_OK ||
        (st = make_store_map_2d(&g.out_map[1], g.k_out, d, s->n_q, d, true)) != FRT_OK ||
        (st = make_store_map_2d(&g.out_map[2], g.v_out, d, s->n_q, d, true)) != FRT_OK)
        return st;
    g.rope = 1;
    fill_rope(s, s->counter, g.ra);
    g.wait_limit_ns = s->wait_limit_ns;
    g.status = s->status_dev;
    cudaError_t e = cudaSuccess;
    if (s->qkv_start) e = cudaEventRecord(s->qkv_start, s->cs);
    if (e == cudaSuccess) e = launch_gemm(g, s->cs);
    if (e == cudaSuccess && s->qkv_stop) e = cudaEventRecord(s->qkv_stop, s->cs);
    if (e != cudaSuccess) return cuda_fail(e, "QKV projection launch");
    s->counter += 1;
    s->phase = kAppended;
    s->last_q = q_buf;
    s->last_k = nullptr;
    s->last_v = nullptr;
    if (slot_out) *slot_out = slot;
    if (evicted_out) *evicted_out = evicted;

    // 2. attention of the chunk (q already rotated), bf16 output for the projection
    if ((st = attention_single(s, q_buf, o_buf, false, 1)) != FRT_OK) return st;

    // 3. output projection
    GemmParams h;
    std::memset(&h, 0, sizeof(h));
    const int bn2 = gemm_block_n_for(s->n_q, d, kEpiPlain, 0);
    if ((st = make_gemm_maps(h, o_buf, w_o, d, s->n_q, d, bn2 / gemm_cluster_m(s->n_q))) != FRT_OK)
        return st;
    h.M = s->n_q;
    h.N = d;
    h.K = d;
    h.epi = kEpiPlain;
    h.c = y;
    h.ldc = d;
    h.c_bf16 = s->cfg.out_dtype == FRT_OUT_BF16;
    if ((st = make_store_map_2d(&h.out_map[0], y, d, s->n_q, d, h.c_bf16 != 0)) != FRT_OK) return st;
    h.wait_limit_ns = s->wait_limit_ns;
    h.status = s->status_dev;
    if (s->proj_start) e = cudaEventRecord(s->proj_start, s->cs);
    if (e == cudaSuccess) e = launch_gemm(h, s->cs);
    if (e == cudaSuccess && s->proj_stop) e = cudaEventRecord(s->proj_stop, s->cs);
    if (e != cudaSuccess) return cuda_fail(e, "output projection launch");
    return FRT_OK;
}

frt_status frt_gemm_plan(int M, int N, int qkv, int d, int* bn, int* ctas) {
    if (!bn || !ctas || M < 1 || N < 1 || (qkv && d < 1))
        return fail(FRT_ERR_INVALID_ARG, "need bn, ctas non-NULL and positive sizes");
    *bn = gemm_block_n_for(M, N, qkv ? kEpiQkv : kEpiPlain, qkv ? d : 0);
    *ctas = gemm_cluster_m(M);
    return FRT_OK;
}

frt_status frt_gemm_bf16(const void* a, const void* b, void* c, int M, int N, int K, int ldc,
                         int c_dtype, void* status, void* cuda_stream) {
    if (!a || !b || !c || !aligned16(a) || !aligned16(b) || !aligned16(c) ||
        (status && (reinterpret_cast<uintptr_t>(status) & 3u)))
        return fail(FRT_ERR_INVALID_ARG, "a, b, c must be non-NULL and 16-byte aligned");
    if (M < 1 || N < 1 || K < 1 || K % 8 != 0 || ldc < N)
        return fail(FRT_ERR_INVALID_ARG, "need M, N, K >= 1, K %% 8 == 0 and ldc >= N");
    if (c_dtype != FRT_OUT_F32 && c_dtype != FRT_OUT_BF16)
        return fail(FRT_ERR_INVALID_ARG, "unknown c_dtype");
    const int esz = c_dtype == FRT_OUT_BF16 ? 2 : 4;
    if ((long long)ldc * esz % 16 != 0)
        return fail(FRT_ERR_INVALID_ARG, "ldc * element size must be a multiple of 16 bytes");
    GemmParams g;
    std::memset(&g, 0, sizeof(g));
    frt_status st;
    if ((st = make_gemm_maps(g, a, b, K, M, N, gemm_block_n_for(M, N, kEpiPlain, 0) / gemm_cluster_m(M))) !=
        FRT_OK)
        return st;
    g.M = M;
    g.N = N;
    g.K = K;
    g.epi = kEpiPlain;
    g.c = c;
    g.ldc = ldc;
    g.c_bf16 = c_dtype == FRT_OUT_BF16;
    if ((st = make_store_map_2d(&g.out_map[0], c, N, M, ldc, g.c_bf16 != 0)) != FRT_OK) return st;
    g.wait_limit_ns = kDefaultWaitLimitNs;
    g.status = static_cast<DeviceStatus*>(status);
    cudaError_t e = launch_gemm(g, static_cast<cudaStream_t>(cuda_stream));
    if (e != cudaSuccess) return cuda_fail(e, "projection launch");
    return FRT_OK;
}

frt_status frt_chunk_step_host(frt_stream_t* s, const void* q_host, const void* k_host,
                               const void* v_host, void* out_host, int* slot_out,
                               long long* evicted_out) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!q_host || !k_host || !v_host || !out_host)
        return fail(FRT_ERR_INVALID_ARG, "NULL host buffer");
    if (s->phase == kRoped) return fail(FRT_ERR_STATE, "a separate rope is pending");
    // Pipelined: kStageSets staging sets are used in turn; the host-to-device copies of
    // this call run on a copy stream while earlier calls' kernels still run, the
    // device-to-host copy on a third stream while later calls compute. Events order each
    // set's reuse: copy-in(n) after compute(n-S), compute(n) after copy-in(n) and after
    // copy-out(n-S), copy-out(n) after compute(n) (S = kStageSets). With three sets a
    // copy may take two kernel steps before compute waits for it: host-device copies
    // on a shared machine run at their full rate most of the time, with occasional slow
    // stretches.
    const size_t in_bytes = s->chunk_elems * 2;
    const size_t out_bytes = s->chunk_elems * (s->cfg.out_dtype == FRT_OUT_BF16 ? 2 : 4);
    const size_t per_set = 3 * in_bytes + out_bytes;
    cudaError_t e;
    if (!s->cp_in) {
        if ((e = cudaStreamCreateWithFlags(&s->cp_in, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaStreamCreateWithFlags(&s->cp_out, cudaStreamNonBlocking)) != cudaSuccess)
            return cuda_fail(e, "copy stream creation");
        for (int b = 0; b < kStageSets; ++b)
            if ((e = cudaEventCreateWithFlags(&s->ev_in[b], cudaEventDisableTiming)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&s->ev_done[b], cudaEventDisableTiming)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&s->ev_out[b], cudaEventDisableTiming)) != cudaSuccess)
                return cuda_fail(e, "event creation");
    }
    if (s->stage_bytes < kStageSets * per_set) {
        if (s->stage) {
            if ((e = cudaDeviceSynchronize()) != cudaSuccess) return cuda_fail(e, "sync");
            cudaFree(s->stage);
            s->stage = nullptr;
            s->stage_bytes = 0;
        }
        if ((e = cudaMalloc(&s->stage, kStageSets * per_set)) != cudaSuccess)
            return cuda_fail(e, "staging");
        s->stage_bytes = kStageSets * per_set;
    }
    const int b = s->stage_turn;
    uint8_t* base = static_cast<uint8_t*>(s->stage) + size_t(b) * per_set;
    void* dq = base;
    void* dk = base + in_bytes;
    void* dv = base + 2 * in_bytes;
    void* dout = base + 3 * in_bytes;
    if ((e = cudaStreamWaitEvent(s->cp_in, s->ev_done[b], 0)) != cudaSuccess ||
        (e = cudaMemcpyAsync(dk, k_host, in_bytes, cudaMemcpyHostToDevice, s->cp_in)) != cudaSuccess ||
        (e = cudaMemcpyAsync(dv, v_host, in_bytes, cudaMemcpyHostToDevice, s->cp_in)) != cudaSuccess ||
        (e = cudaMemcpyAsync(dq, q_host, in_bytes, cudaMemcpyHostToDevice, s->cp_in)) != cudaSuccess ||
        (e = cudaEventRecord(s->ev_in[b], s->cp_in)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(s->cs, s->ev_in[b], 0)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(s->cs, s->ev_out[b], 0)) != cudaSuccess)
        return cuda_fail(e, "host-to-device copy");
    if ((st = frt_chunk_step(s, dq, dk, dv, dout, slot_out, evicted_out)) != FRT_OK) return st;
    if ((e = cudaEventRecord(s->ev_done[b], s->cs)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(s->cp_out, s->ev_done[b], 0)) != cudaSuccess ||
        (e = cudaMemcpyAsync(out_host, dout, out_bytes, cudaMemcpyDeviceToHost, s->cp_out)) !=
            cudaSuccess ||
        (e = cudaEventRecord(s->ev_out[b], s->cp_out)) != cudaSuccess)
        return cuda_fail(e, "device-to-host copy");
    s->stage_turn = (s->stage_turn + 1) % kStageSets;
    return FRT_OK;
}

frt_status frt_attention_plan(int n, const int* n_q, const long long* n_kv, int heads, int sms,
                              int* n_full, int* n_split) {
    if (n < 1 || !n_q || !n_kv || heads < 1 || !n_full || !n_split)
        return fail(FRT_ERR_INVALID_ARG, "need n >= 1, heads >= 1 and non-NULL arrays");
    std::vector<int> tiles;
    std::vector<unsigned char> single;
    for (int i = 0; i < n; ++i) {
        if (n_q[i] < 1 || n_kv[i] < 1) return fail(FRT_ERR_INVALID_ARG, "sizes must be >= 1");
        stream_groups(n_q[i], heads, n_kv[i], tiles, single);
    }
    const SplitPlan pl = plan_attention(tiles.data(), single.data(), int(tiles.size()),
                                        sms > 0 ? sms : num_sms(), kMaxSplit, -1, -1);
    *n_full = pl.n_full;
    *n_split = pl.n_split;
    return FRT_OK;
}

frt_status frt_chunk_attention_batched(frt_stream_t* const* streams, int n, const void* const* q,
                                       void* const* out) {
    if (!streams || !q || !out || n < 1 || n > kMaxBatchStreams)
        return fail(FRT_ERR_INVALID_ARG, "need 1 <= n <= %d streams and q/out arrays",
                    kMaxBatchStreams);
    frt_stream_t* s0 = streams[0];
    frt_status st;
    for (int i = 0; i < n; ++i) {
        frt_stream_t* s = streams[i];
        if ((st = require_configured(s)) != FRT_OK) return st;
        if (s->heads != s0->heads || s->head_dim != s0->head_dim || s->scale != s0->scale ||
            s->cfg.out_dtype != s0->cfg.out_dtype)
            return fail(FRT_ERR_UNSUPPORTED, "batched streams must share heads, head_dim, scale, dtype");
        if (s->phase != kAppended) return fail(FRT_ERR_STATE, "stream %d has not appended", i);
        if (!q[i] || !out[i] || !aligned16(q[i]) || !aligned16(out[i]))
            return fail(FRT_ERR_INVALID_ARG, "q/out %d NULL or misaligned", i);
        if (q[i] != s->last_q) return fail(FRT_ERR_STATE, "q %d is not this chunk's rotated q", i);
        for (int j = 0; j < i; ++j)
            if (streams[j] == s) return fail(FRT_ERR_INVALID_ARG, "stream %d repeated", i);
    }
    // longest KV first (LPT): items are handed to SMs in launch order
    std::vector<int> order(n);
    for (int i = 0; i < n; ++i) order[i] = i;
    auto n_kv = [&](int i) {
        return std::min<long long>(streams[i]->counter, streams[i]->window) * streams[i]->n_q;
    };
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return n_kv(a) > n_kv(b); });
    auto* p = new (std::nothrow) AttnParams<kMaxBatchStreams>();
    if (!p) return fail(FRT_ERR_OOM, "host allocation failed");
    std::memset(p, 0, sizeof(*p));
    // query groups in launch order (streams longest KV first, then head-major) and the
    // work split of the launch
    std::vector<int> tiles;
    std::vector<unsigned char> single;
    for (int oi = 0; oi < n; ++oi) {
        const int i = order[oi];
        stream_groups(streams[i]->n_q, streams[i]->heads, n_kv(i), tiles, single);
    }
    const long long groups_total = (long long)tiles.size();
    const SplitPlan pl = plan_attention(tiles.data(), single.data(), int(groups_total), num_sms(),
                                        kMaxSplit, -1, -1);
    if ((st = ensure_scratch(s0, plan_rows(pl, groups_total), plan_tails(pl, groups_total))) !=
        FRT_OK) {
        delete p;
        return st;
    }
    p->n_full = pl.n_full;
    p->n_split = pl.n_split;
    if (pl.n_split > 1 &&
        (st = make_part_map(&p->part_map, s0->part_o, s0->head_dim, s0->part_rows)) != FRT_OK) {
        delete p;
        return st;
    }
    p->part_o = s0->part_o;
    p->part_ml = s0->part_ml;
    p->counters = s0->counters;
    p->groups_total = int(groups_total);
    p->part_rows_cap = s0->part_rows;
    p->tails_cap = s0->part_tails;
    int groups = 0;
    for (int oi = 0; oi < n; ++oi) {
        const int i = order[oi];
        frt_stream_t* s = streams[i];
        AttnStreamDesc& d = p->s[oi];
        const long long nkv = n_kv(i);
        if ((st = make_map(&d.q_map, q[i], s->head_dim, s->heads, s->n_q)) != FRT_OK ||
            (st = make_map(&d.k_map, s->cache_k, s->head_dim, s->heads, nkv)) != FRT_OK ||
            (st = make_map(&d.v_map, s->cache_v, s->head_dim, s->heads, nkv)) != FRT_OK) {
            delete p;
            return st;
        }
        if ((st = make_out_map(&d.out_map, out[i], s->head_dim, s->heads, s->n_q,
                               s0->cfg.out_dtype == FRT_OUT_BF16)) != FRT_OK) {
            delete p;
            return st;
        }
        d.out = out[i];
        d.n_q = s->n_q;
        d.n_kv = int(nkv);
        d.n_qpairs = (s->n_q + 255) / 256;
        d.group_begin = groups;
        groups += d.n_qpairs * s->heads;
    }
    const int items = int(pl.n_full + (groups_total - pl.n_full) * pl.n_split);
    p->n_streams = n;
    p->heads = s0->heads;
    p->total_items = items;
    p->out_bf16 = s0->cfg.out_dtype == FRT_OUT_BF16;
    p->scale_log2 = float(double(s0->scale) * 1.4426950408889634);
    p->wait_limit_ns = s0->wait_limit_ns;
    p->status = s0->status_dev;
    cudaError_t e = cudaSuccess;
    for (int i = 1; i < n && e == cudaSuccess; ++i)
        if (streams[i]->cs != s0->cs) {
            e = cudaEventRecord(streams[i]->ev, streams[i]->cs);
            if (e == cudaSuccess) e = cudaStreamWaitEvent(s0->cs, streams[i]->ev, 0);
        }
    if (e == cudaSuccess && s0->attn_start) e = cudaEventRecord(s0->attn_start, s0->cs);
    if (e == cudaSuccess) e = launch_attention_batched(*p, s0->head_dim, s0->cs);
    if (e == cudaSuccess && s0->attn_stop) e = cudaEventRecord(s0->attn_stop, s0->cs);
    delete p;
    if (e != cudaSuccess) return cuda_fail(e, "batched attention launch");
    bool other = false;
    for (int i = 1; i < n; ++i) other |= streams[i]->cs != s0->cs;
    if (other) {
        if ((e = cudaEventRecord(s0->ev, s0->cs)) != cudaSuccess) return cuda_fail(e, "event");
        for (int i = 1; i < n; ++i)
            if (streams[i]->cs != s0->cs &&
                (e = cudaStreamWaitEvent(streams[i]->cs, s0->ev, 0)) != cudaSuccess)
                return cuda_fail(e, "event wait");
    }
    return FRT_OK;
}

frt_status frt_stream_sync(frt_stream_t* s) {
    if (!s) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if (!s->configured) return FRT_OK;
    cudaError_t e = cudaStreamSynchronize(s->cs);
    if (e == cudaSuccess && s->cp_in) e = cudaStreamSynchronize(s->cp_in);
    if (e == cudaSuccess && s->cp_out) e = cudaStreamSynchronize(s->cp_out);
    if (e != cudaSuccess) return cuda_fail(e, "stream sync");
    frt_status st = check_device_status(s);
    // the debug build also compares the guard words around the cache at every sync
    if (st == FRT_OK && kDebugBuild) st = frt_stream_check_guards(s);
    return st;
}

frt_status frt_stream_reset(frt_stream_t* s) {
    if (!s) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if (!s->configured) return fail(FRT_ERR_STATE, "stream not configured");
    cudaError_t e = cudaStreamSynchronize(s->cs);
    if (e == cudaSuccess && s->cp_in) e = cudaStreamSynchronize(s->cp_in);
    if (e == cudaSuccess && s->cp_out) e = cudaStreamSynchronize(s->cp_out);
    if (e != cudaSuccess) return cuda_fail(e, "stream sync");
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    // the merge counters too: a launch that gave up part-way (the usual reason for a
    // reset) may have left some of them counted, which would elect a merging split early
    if ((e = cudaMemsetAsync(s->cache_k, 0, cache_bytes, s->cs)) != cudaSuccess ||
        (e = cudaMemsetAsync(s->cache_v, 0, cache_bytes, s->cs)) != cudaSuccess ||
        (s->counters && (e = cudaMemsetAsync(s->counters, 0, size_t(s->part_tails) * sizeof(int),
                                             s->cs)) != cudaSuccess) ||
        (e = cudaStreamSynchronize(s->cs)) != cudaSuccess)
        return cuda_fail(e, "cache clear");
    std::memset(s->status_host, 0, sizeof(DeviceStatus));
    s->counter = 0;
    s->phase = kStart;
    s->last_q = s->last_k = s->last_v = nullptr;
    return FRT_OK;
}

void frt_stream_destroy(frt_stream_t* s) {
    if (!s) return;
    // device memory may exist without a completed configure (one that failed part-way)
    if (s->configured || s->cache_k || s->stage) cudaStreamSynchronize(s->cs);
    free_device(s);
    delete s;
}

frt_status frt_stream_set_block_events(frt_stream_t* s, void* qkv_start, void* qkv_stop,
                                       void* out_start, void* out_stop) {
    if (s == nullptr) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    s->qkv_start = static_cast<cudaEvent_t>(qkv_start);
    s->qkv_stop = static_cast<cudaEvent_t>(qkv_stop);
    s->proj_start = static_cast<cudaEvent_t>(out_start);
    s->proj_stop = static_cast<cudaEvent_t>(out_stop);
    return FRT_OK;
}

long long frt_stream_chunk_counter(const frt_stream_t* s) { return s ? s->counter : -1; }

frt_status frt_stream_set_attention_events(frt_stream_t* s, void* start_event,
                                           void* stop_event) {
    if (!s) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if ((start_event == nullptr) != (stop_event == nullptr))
        return fail(FRT_ERR_INVALID_ARG, "give both events or neither");
    s->attn_start = static_cast<cudaEvent_t>(start_event);
    s->attn_stop = static_cast<cudaEvent_t>(stop_event);
    return FRT_OK;
}

frt_status frt_stream_set_append_events(frt_stream_t* s, void* start_event, void* stop_event) {
    if (!s) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if ((start_event == nullptr) != (stop_event == nullptr))
        return fail(FRT_ERR_INVALID_ARG, "give both events or neither");
    s->app_start = static_cast<cudaEvent_t>(start_event);
    s->app_stop = static_cast<cudaEvent_t>(stop_event);
    return FRT_OK;
}

int frt_debug_build(void) { return kDebugBuild ? 1 : 0; }

frt_status frt_stream_check_guards(frt_stream_t* s) {
    if (!s) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if (!s->configured || !s->alloc_k) return fail(FRT_ERR_STATE, "stream not configured");
    cudaError_t e = cudaStreamSynchronize(s->cs);
    if (e != cudaSuccess) return cuda_fail(e, "stream sync");
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    std::vector<unsigned char> h(std::max(kGuardBytes, s->rear_bytes));
    const char* names[2] = {"K", "V"};
    unsigned char* allocs[2] = {s->alloc_k, s->alloc_v};
    for (int b = 0; b < 2; ++b) {
        const struct { size_t off, len; const char* where; } parts[2] = {
            {0, kGuardBytes, "before"}, {kGuardBytes + cache_bytes, s->rear_bytes, "after"}};
        for (const auto& pt : parts) {
            if ((e = cudaMemcpy(h.data(), allocs[b] + pt.off, pt.len, cudaMemcpyDeviceToHost)) !=
                cudaSuccess)
                return cuda_fail(e, "guard read");
            for (size_t i = 0; i < pt.len; ++i)
                if (h[i] != kGuardByte)
                    return fail(FRT_ERR_BOUNDS, "guard word %s the %s cache overwritten (byte %zu)",
                                pt.where, names[b], i);
        }
    }
    return FRT_OK;
}

frt_status frt_stream_save(frt_stream_t* s, void* k_dst, void* v_dst, long long* counter) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!k_dst || !v_dst || !counter) return fail(FRT_ERR_INVALID_ARG, "NULL destination");
    if (s->phase == kRoped) return fail(FRT_ERR_STATE, "a chunk is half done (rope without append)");
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    cudaError_t e;
    if ((e = cudaMemcpyAsync(k_dst, s->cache_k, cache_bytes, cudaMemcpyDefault, s->cs)) !=
            cudaSuccess ||
        (e = cudaMemcpyAsync(v_dst, s->cache_v, cache_bytes, cudaMemcpyDefault, s->cs)) !=
            cudaSuccess)
        return cuda_fail(e, "snapshot copy");
    *counter = s->counter;
    return FRT_OK;
}

frt_status frt_stream_restore(frt_stream_t* s, const void* k_src, const void* v_src,
                              long long counter) {
    frt_status st = require_configured(s);
    if (st != FRT_OK) return st;
    if (!k_src || !v_src) return fail(FRT_ERR_INVALID_ARG, "NULL source");
    if (counter < 0) return fail(FRT_ERR_INVALID_ARG, "counter must be >= 0");
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    cudaError_t e;
    if ((e = cudaMemcpyAsync(s->cache_k, k_src, cache_bytes, cudaMemcpyDefault, s->cs)) !=
            cudaSuccess ||
        (e = cudaMemcpyAsync(s->cache_v, v_src, cache_bytes, cudaMemcpyDefault, s->cs)) !=
            cudaSuccess)
        return cuda_fail(e, "restore copy");
    s->counter = counter;
    s->phase = kStart;
    s->last_q = s->last_k = s->last_v = nullptr;
    return FRT_OK;
}

frt_status frt_stream_cache(const frt_stream_t* s, const void** k_cache, const void** v_cache,
                            long long* rows) {
    if (!s) return fail(FRT_ERR_INVALID_ARG, "NULL stream handle");
    if (!s->configured) return fail(FRT_ERR_STATE, "stream not configured");
    if (k_cache) *k_cache = s->cache_k;
    if (v_cache) *v_cache = s->cache_v;
    if (rows) *rows = (long long)s->window * s->n_q;
    return FRT_OK;
}

}  // extern "C"

void frt::set_last_error(const char* msg) { g_last_error = msg; }

// Device pointer of a stream's status block (used by the self-test entry points).
extern "C" void* frt_internal_status_dev(frt_stream_t* s) {
    return (s && s->configured) ? static_cast<void*>(s->status_dev) : nullptr;
}

// ---------------------------------------------------------------------------------------
// Per-denoising-step caches: a group of independent streams advanced by pipeline ticks.
// ---------------------------------------------------------------------------------------
struct frt_steps {
    int n = 0;
    frt_stream_t* st[kMaxBatchStreams] = {};
};

extern "C" {

frt_steps_t* frt_steps_create(int n_steps, int heads, int head_dim, int tokens_per_frame,
                              int frames_per_chunk, int window_chunks) {
    if (n_steps < 1 || n_steps > kMaxBatchStreams) {
        fail(FRT_ERR_INVALID_ARG, "1 <= n_steps <= %d", kMaxBatchStreams);
        return nullptr;
    }
    frt_steps_t* g = new (std::nothrow) frt_steps();
    if (!g) {
        fail(FRT_ERR_OOM, "host allocation failed");
        return nullptr;
    }
    for (int i = 0; i < n_steps; ++i) {
        g->st[i] = frt_stream_create(heads, head_dim, tokens_per_frame, frames_per_chunk,
                                     window_chunks);
        if (!g->st[i]) {
            frt_steps_destroy(g);
            return nullptr;   // frt_last_error() set by frt_stream_create
        }
        g->n = i + 1;
    }
    return g;
}

frt_status frt_steps_configure(frt_steps_t* g, const frt_config* cfg) {
    if (!g || !cfg) return fail(FRT_ERR_INVALID_ARG, "NULL argument");
    for (int i = 0; i < g->n; ++i) {
        frt_status st = frt_stream_configure(g->st[i], cfg);
        if (st != FRT_OK) return st;
    }
    return FRT_OK;
}

frt_stream_t* frt_steps_stream(const frt_steps_t* g, int step) {
    if (!g || step < 0 || step >= g->n) return nullptr;
    return g->st[step];
}

frt_status frt_steps_tick(frt_steps_t* g, unsigned int active_mask, void* const* q,
                          void* const* k, const void* const* v, void* const* out) {
    if (!g || !q || !k || !v || !out) return fail(FRT_ERR_INVALID_ARG, "NULL argument");
    if (active_mask == 0) return FRT_OK;
    if (g->n < 32 && (active_mask >> g->n) != 0)
        return fail(FRT_ERR_INVALID_ARG, "active_mask names a step beyond n_steps");
    frt_stream_t* streams[kMaxBatchStreams];
    const void* qs[kMaxBatchStreams];
    void* outs[kMaxBatchStreams];
    int n = 0;
    frt_status st;
    for (int i = 0; i < g->n; ++i) {
        if (!((active_mask >> i) & 1u)) continue;
        if ((st = frt_rope3d_qk(g->st[i], q[i], k[i])) != FRT_OK) return st;
        if ((st = frt_kv_append_evict(g->st[i], k[i], v[i], nullptr, nullptr)) != FRT_OK) return st;
        streams[n] = g->st[i];
        qs[n] = q[i];
        outs[n] = out[i];
        ++n;
    }
    return frt_chunk_attention_batched(streams, n, qs, outs);
}

void frt_steps_destroy(frt_steps_t* g) {
    if (!g) return;
    for (int i = 0; i < g->n; ++i) frt_stream_destroy(g->st[i]);
    delete g;
}

}  // extern "C"

extern "C" frt_status frt_selftest_append_past_ring(void) {
#ifdef FRT_DEBUG
    g_append_past_ring = 1;
    return FRT_OK;
#else
    return fail(FRT_ERR_UNSUPPORTED, "only the FRT_DEBUG build has this hook");
#endif
}

extern "C" frt_status frt_selftest_poke_guard(frt_stream_t* s, int which) {
    if (!s || !s->configured || !s->alloc_k) return fail(FRT_ERR_STATE, "stream not configured");
    if (which < 0 || which > 3) return fail(FRT_ERR_INVALID_ARG, "which in 0..3");
    const size_t cache_bytes = size_t(s->window) * s->chunk_elems * 2;
    unsigned char* a = (which & 1) ? s->alloc_v : s->alloc_k;
    unsigned char* at = (which & 2) ? a + kGuardBytes + cache_bytes : a + kGuardBytes - 1;
    cudaError_t e = cudaStreamSynchronize(s->cs);
    if (e == cudaSuccess) e = cudaMemset(at, 0x00, 1);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "guard poke");
    return FRT_OK;
}
