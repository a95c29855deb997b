// frt_noalloc.cu — chunk attention for callers that cannot allocate device memory.
//
// Some callers may not call cudaMalloc at all: code running under a memory planner or
// arena that owns every device byte, real-time loops where an allocation (which can
// synchronise the device) is not allowed, or integrations whose only device memory is
// the buffers they pass in. frt_chunk_attention_noalloc serves them: it runs the same
// split-KV attention kernel as frt_chunk_attention over caller-owned q/K/V/out, and the
// kernel's only scratch (split partials and merge counters) lives in the file-scope array
// below, which every GPU that loads this library holds until the process exits.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <utility>
#include <vector>

#include "../../include/frt.h"
#include "frt_internal.h"

using namespace frt;

namespace {

// Static scratch: partial rows (unnormalised O, fp32) + (max, sum) per row + one merge
// counter per query group. 8 MiB + 128 KiB + 16 KiB.
constexpr size_t kPartBytes = size_t(8) << 20;               // partial O rows
constexpr size_t kMlBytes = size_t(16384) * sizeof(float2);   // (max, sum) rows
constexpr int kMaxGroups = 4096;                              // query groups (heads x 256 rows)
constexpr size_t kScratchBytes = kPartBytes + kMlBytes + size_t(kMaxGroups) * sizeof(int);

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// Device address of g_noalloc_scratch per CUDA context. A __device__ symbol's address
// belongs to the context that loaded the module, so the cache is keyed by the context's
// unique ID (cuCtxGetId: never reused within a process), not by the device ordinal: a
// non-primary context, or the new primary context after a cudaDeviceReset, looks the
// address up again instead of using a stale one.
std::mutex g_mu;
std::vector<std::pair<unsigned long long, void*>> g_scratch_by_ctx;

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

template <typename Fn>
Fn driver_fn(const char* name) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
        return reinterpret_cast<Fn>(p);
    return nullptr;
}

// Unique ID of the calling thread's current context; 0 if none is current or the driver
// does not offer the query.
unsigned long long current_ctx_id() {
    static CtxGetCurrentFn get_cur = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        get_cur = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
        get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
    });
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (!get_cur || !get_id || get_cur(&ctx) != CUDA_SUCCESS || ctx == nullptr ||
        get_id(ctx, &id) != CUDA_SUCCESS)
        return 0;
    return id;
}

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

// q/K/V: 3D (head_dim, heads, rows) bf16, box (64, 1, 128), 128-byte swizzle.
bool encode(CUtensorMap* map, const void* base, int head_dim, int heads, long long rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {cuuint64_t(head_dim), cuuint64_t(heads), cuuint64_t(rows)};
    cuuint64_t strides[2] = {cuuint64_t(head_dim) * 2, cuuint64_t(heads) * head_dim * 2};
    cuuint32_t box[3] = {64, 1, 128};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// Output [rows, heads, head_dim] fp32 or bf16 for TMA stores: box of 128 bytes of head_dim
// x 1 head x 128 rows, 128-byte swizzle.
bool encode_out(CUtensorMap* map, void* base, int head_dim, int heads, long long rows, bool bf16) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const int es = bf16 ? 2 : 4;
    cuuint64_t dims[3] = {cuuint64_t(head_dim), cuuint64_t(heads), cuuint64_t(rows)};
    cuuint64_t strides[2] = {cuuint64_t(head_dim) * es, cuuint64_t(heads) * head_dim * es};
    cuuint32_t box[3] = {cuuint32_t(128 / es), 1, 128};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3,
              base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Split-KV partial rows [rows, head_dim] fp32: box 32 x 128, 128-byte swizzle.
bool encode_part(CUtensorMap* map, float* base, int head_dim, long long rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {cuuint64_t(head_dim), cuuint64_t(rows)};
    cuuint64_t strides[1] = {cuuint64_t(head_dim) * 4};
    cuuint32_t box[2] = {32, 128};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

frt_status fail(frt_status st, const char* msg) {
    set_last_error(msg);
    return st;
}
// A CUDA runtime call of this entry point failed (see clear_cuda_error).
frt_status cuda_failed(const char* msg) {
    clear_cuda_error();
    return fail(FRT_ERR_CUDA, msg);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" frt_status frt_chunk_attention_noalloc(const void* q, const void* k, const void* v,
                                                  void* out, int n_q, int n_kv, int heads,
                                                  int head_dim, double sm_scale, int out_dtype,
                                                  void* status, void* cuda_stream) {
    if (!q || !k || !v || !out || !aligned16(q) || !aligned16(k) || !aligned16(v) ||
        !aligned16(out) || (status && (reinterpret_cast<uintptr_t>(status) & 3u)))
        return fail(FRT_ERR_INVALID_ARG, "q, k, v, out must be non-NULL and 16-byte aligned");
    if (n_q < 1 || n_kv < 1 || heads < 1 || heads > 1024 || n_q > (1 << 20) || n_kv > (1 << 24))
        return fail(FRT_ERR_INVALID_ARG, "bad n_q, n_kv or heads");
    if (head_dim != 64 && head_dim != 128)
        return fail(FRT_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (out_dtype != FRT_OUT_F32 && out_dtype != FRT_OUT_BF16)
        return fail(FRT_ERR_INVALID_ARG, "unknown out_dtype");
    const int n_qpairs = (n_q + 255) / 256;
    const long long groups = (long long)n_qpairs * heads;
    if (groups > kMaxGroups)
        return fail(FRT_ERR_UNSUPPORTED,
                    "heads * ceil(n_q / 256) exceeds the static maximum of 4096 query groups; "
                    "use frt_chunk_attention for larger chunks");

    // one-time set-up per context: the array's device address (host code may not use
    // the symbol itself as a device pointer). The look-up also makes the device's primary
    // context current when the calling thread has none yet.
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_failed("no usable current device");
    void* base = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        unsigned long long ctx = current_ctx_id();
        for (const auto& entry : g_scratch_by_ctx)
            if (ctx != 0 && entry.first == ctx) base = entry.second;
        if (!base) {
            e = cudaGetSymbolAddress(&base, g_noalloc_scratch);
            if (e != cudaSuccess || !base)
                return cuda_failed("cudaGetSymbolAddress of the static scratch failed");
            if (ctx == 0) ctx = current_ctx_id();
            if (ctx == 0) return fail(FRT_ERR_CUDA, "no current CUDA context after set-up");
            g_scratch_by_ctx.emplace_back(ctx, base);
        }
    }
    uint8_t* b = static_cast<uint8_t*>(base);
    float* part_o = reinterpret_cast<float*>(b);
    float2* part_ml = reinterpret_cast<float2*>(b + kPartBytes);
    int* counters = reinterpret_cast<int*>(b + kPartBytes + kMlBytes);

    // largest useful split whose partials fit the static buffer (split 1 needs none)
    const long long sms = num_sms();
    const int tiles = (n_kv + 127) / 128;
    const size_t cap_rows = std::min(kPartBytes / (size_t(head_dim) * 4), kMlBytes / sizeof(float2));
    int split = 1;
    double best = double((groups + sms - 1) / sms);
    for (int sp = 2; sp <= kMaxSplit && tiles >= 2 * sp; ++sp) {
        if (size_t(groups) * sp * 256 > cap_rows) break;
        const double t = double((groups * sp + sms - 1) / sms) / sp * (1.0 + 0.02 * (sp - 1));
        if (t < best - 1e-9) {
            best = t;
            split = sp;
        }
    }

    AttnParams<1> p;
    std::memset(&p, 0, sizeof(p));
    AttnStreamDesc& d = p.s[0];
    if (!encode(&d.q_map, q, head_dim, heads, n_q) || !encode(&d.k_map, k, head_dim, heads, n_kv) ||
        !encode(&d.v_map, v, head_dim, heads, n_kv))
        return fail(FRT_ERR_CUDA, "tensor map encoding failed");
    if (!encode_out(&d.out_map, out, head_dim, heads, n_q, out_dtype == FRT_OUT_BF16) ||
        (split > 1 && !encode_part(&p.part_map, part_o, head_dim, (long long)groups * split * 256)))
        return fail(FRT_ERR_CUDA, "tensor map encoding failed");
    d.out = out;
    d.n_q = n_q;
    d.n_kv = n_kv;
    d.n_qpairs = n_qpairs;
    p.n_streams = 1;
    p.heads = heads;
    p.n_full = 0;          // every group is cut into `split` parts (split 1: run whole)
    p.n_split = split;
    p.groups_total = int(groups);
    p.part_rows_cap = (long long)cap_rows;
    p.tails_cap = kMaxGroups;
    p.total_items = int(groups * split);
    p.part_o = part_o;
    p.part_ml = part_ml;
    p.counters = counters;
    p.out_bf16 = out_dtype == FRT_OUT_BF16;
    const double scale = sm_scale > 0 ? sm_scale : 1.0 / std::sqrt(double(head_dim));
    p.scale_log2 = float(scale * 1.4426950408889634);
    p.wait_limit_ns = 2000000000ull;
    p.status = static_cast<DeviceStatus*>(status);
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    // merge counters must start at zero: clear this call's share of the shared array
    if (split > 1 &&
        (e = cudaMemsetAsync(counters, 0, size_t(groups) * sizeof(int), st)) != cudaSuccess)
        return cuda_failed("clearing the merge counters failed");
    if ((e = launch_attention_single(p, head_dim, false, st)) != cudaSuccess)
        return cuda_failed(cudaGetErrorString(e));
    return FRT_OK;
}
