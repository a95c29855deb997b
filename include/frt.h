/*
 * frt.h — C ABI of the GB300 (sm_103a) streaming frame-chunk attention library.
 *
 * The workload is the per-chunk attention of an autoregressive video
 * diffusion transformer over a persistent, rolling KV cache: the cache is the
 * cross-batch state that batch j inherits from batch j-1 (arxiv 2607.18171,
 * section 2 "Problem Formulation", the lambda = 1 state edge; Appendix A.1.2
 * "Pipeline graph"), inputs arrive as frame chunks (Appendix A.1.1), and each
 * denoising step owns an independent cache (section 3.1 "Case study";
 * Appendix A.4), which here is one frt_stream_t per (request, step).
 *
 * One chunk c of a stream runs three operations, in this order:
 *   1. 3D rotary embedding of q and k at the chunk's positions   (frt_rope3d_qk)
 *   2. append of (k, v) to ring slot c mod W, evicting chunk c-W  (frt_kv_append_evict)
 *   3. attention of the chunk's queries over every cached key     (frt_chunk_attention)
 * or all three at once with frt_chunk_step (RoPE-Q runs inside the attention
 * kernel's prologue, RoPE-K inside the append).
 *
 * Tensors: token-major [tokens, heads, head_dim], contiguous, bf16 for q/k/v,
 * fp32 or bf16 for out, device pointers (unless a name ends in _host),
 * 16-byte aligned. Token i of a chunk is frame i / (grid_h*grid_w), row
 * (i mod grid_h*grid_w) / grid_w, column i mod grid_w.
 *
 * Ownership: the caller owns q/k/v/out; a stream owns its KV cache (allocated
 * in frt_stream_configure, freed in frt_stream_destroy). A handle is not
 * thread-safe; distinct handles are independent.
 *
 * Asynchrony: every call enqueues work on the stream's configured CUDA stream
 * and returns after launch. Host-side argument and state errors are returned
 * immediately and enqueue nothing. Device-side errors (a bounded wait that gave
 * up) are recorded in a per-stream status word and returned by
 * frt_stream_sync or by the next call on the stream.
 */
#ifndef FRT_H
#define FRT_H

#ifdef __cplusplus
extern "C" {
#endif

typedef struct frt_stream frt_stream_t; /* opaque; owns its KV cache */

typedef enum frt_status {
    FRT_OK = 0,
    FRT_ERR_INVALID_ARG = 1,  /* NULL/misaligned pointer, bad size or config */
    FRT_ERR_STATE = 2,        /* call out of the rope -> append -> attention order */
    FRT_ERR_OOM = 3,          /* device or pinned allocation failed */
    FRT_ERR_CUDA = 4,         /* a CUDA runtime/driver call failed */
    FRT_ERR_UNSUPPORTED = 5,  /* head_dim or shape the kernels do not handle */
    FRT_ERR_TIMEOUT = 6,      /* a device-side bounded wait gave up */
    FRT_ERR_BOUNDS = 7        /* a guard word around the KV cache was overwritten, or (debug
                                 build) a kernel's bounds check refused an access */
} frt_status;

typedef enum frt_out_dtype { FRT_OUT_F32 = 0, FRT_OUT_BF16 = 1 } frt_out_dtype;

/* Per-stream configuration (frt_stream_configure). */
typedef struct frt_config {
    int grid_h, grid_w;            /* latent grid; grid_h * grid_w == tokens_per_frame */
    int rope_dt, rope_dh, rope_dw; /* head_dim split [t | h | w]; each even, sum == head_dim */
    double theta;                  /* RoPE base (10000) */
    double sm_scale;               /* softmax scale; <= 0 selects 1/sqrt(head_dim) */
    int out_dtype;                 /* frt_out_dtype */
    void* cuda_stream;             /* cudaStream_t all work is enqueued on; NULL = legacy stream */
} frt_config;

/* Create a stream handle: one (video stream, denoising step) and its persistent KV
 * cache, the cross-batch state that batch j inherits from batch j-1 (paper section 2
 * "Problem Formulation", the lambda = 1 edge; Appendix A.1.2 "Pipeline graph"); chunks
 * of frames_per_chunk frames are the batches (Appendix A.1.1 "Initial assumptions").
 *   heads >= 1; head_dim in {64, 128}; heads * head_dim <= 12800; tokens_per_frame >= 1;
 *   frames_per_chunk >= 1; window_chunks >= 1 (the window counts the current chunk).
 * Nq = frames_per_chunk * tokens_per_frame must be <= 2^20 and
 * window_chunks * Nq <= 2^24. Allocates no device memory.
 * Returns NULL on error; frt_last_error() then describes it. */
frt_stream_t* frt_stream_create(int heads, int head_dim, int tokens_per_frame,
                                int frames_per_chunk, int window_chunks);

/* Fill *cfg with the defaults for s: grid 1 x tokens_per_frame, RoPE split
 * (D/4, 3D/8, 3D/8) rounded to even, theta 10000, sm_scale 1/sqrt(D), fp32
 * output, legacy CUDA stream. */
frt_status frt_config_default(const frt_stream_t* s, frt_config* cfg);

/* Validate and apply *cfg; allocates (once) and zero-fills the KV cache
 * (2 * window_chunks * Nq * heads * head_dim bf16) and the RoPE tables, and
 * resets the chunk counter to 0. Synchronous. Must precede every other call.
 * A configure that fails after validation leaves the stream unconfigured: later
 * calls return FRT_ERR_STATE until a configure succeeds. */
frt_status frt_stream_configure(frt_stream_t* s, const frt_config* cfg);

/* Operation 1 (the paper does not define the position encoding: it deploys video DiTs,
 * sections 4.3.3-4.3.4, whose attention runs on rotated q and k; the segment split and
 * pairing are this library's convention, fixed by frt_config):
 * rotate q and k (bf16 [Nq, heads, head_dim]) in place at the
 * positions of chunk c = frt_stream_chunk_counter(s): token i sits at
 * (t = c * frames_per_chunk + i / tokens_per_frame, row, column); in segment
 * a of width d_a, pair (2j, 2j+1) turns by pos_a * theta^(-2j/d_a).
 * Allowed at the start of a chunk (after configure/reset, an append, or an
 * attention); otherwise FRT_ERR_STATE. */
frt_status frt_rope3d_qk(frt_stream_t* s, void* q, void* k);

/* Operation 2, the write side of the KV-cache state edge (section 2 "Problem
 * Formulation"; section 3.2 "IR design": a node's persistent-state writes; Appendix
 * A.1.2: the cache batch j+1 inherits from batch j): copy the rotated k and v of chunk
 * c into ring slot c mod W
 * (cache rows [slot*Nq, (slot+1)*Nq)), overwriting evicted chunk c - W, then
 * advance the counter. *slot_out = c mod W, *evicted_out = c - W or -1 (either
 * pointer may be NULL). Indices are computed on the host (exact). Must follow
 * frt_rope3d_qk of the same chunk; otherwise FRT_ERR_STATE. */
frt_status frt_kv_append_evict(frt_stream_t* s, const void* k, const void* v,
                               int* slot_out, long long* evicted_out);

/* Operation 3, the read side of that state edge inside the DiT, the stage that sets the
 * pipelines' frame-rate ceiling (Appendix B.1 "What drives the tradeoff"):
 * out[i, h, :] = sum_j softmax_j(sm_scale * <q[i,h], K[j,h]>) V[j,h,:]
 * over every valid cached row j (n_c * Nq rows, n_c = min(c + 1, W) for the
 * chunk c just appended): bidirectional inside the chunk, all earlier chunks
 * of the window. bf16 operands, fp32 accumulation, P rounded to bf16 for the
 * PV product. q must be the pointer rotated by the last frt_rope3d_qk; k and v
 * must be the pointers of the last append, or NULL (K/V are read from the
 * cache either way). out: [Nq, heads, head_dim] in the configured dtype.
 * Must follow an append; otherwise FRT_ERR_STATE. */
frt_status frt_chunk_attention(const void* q, const void* k, const void* v,
                               void* out, frt_stream_t* s);

/* Operations 1-3 fused for one chunk (one batch's pass over the state edge of section 2
 * and Appendix A.1.2): q, k, v are the raw (unrotated) inputs
 * and are not modified; RoPE-K runs inside the append (rotated K goes to the
 * cache only) and RoPE-Q inside the attention kernel's prologue. Same result
 * as the three separate calls. Allowed at the start of a chunk. */
frt_status frt_chunk_step(frt_stream_t* s, const void* q, const void* k,
                          const void* v, void* out, int* slot_out,
                          long long* evicted_out);

/* frt_chunk_step with HOST buffers: copies q, k, v host -> device into
 * stream-owned staging buffers, runs the fused step, copies out device ->
 * host. Consecutive calls are pipelined: three staging sets are used in turn,
 * the copies in run on an internal copy stream while earlier calls' kernels run,
 * and the copy out on another while later calls compute (events keep every set's
 * reuse ordered). Host buffers must stay valid, and out_host unread, until
 * frt_stream_sync returns (pinned memory makes the copies asynchronous). The
 * staging (3 x (3 inputs + output)) is allocated on the first call. */
frt_status frt_chunk_step_host(frt_stream_t* s, const void* q_host,
                               const void* k_host, const void* v_host,
                               void* out_host, int* slot_out,
                               long long* evicted_out);

/* The attention slice of one DiT block for chunk c: QKV projection -> 3D RoPE
 * -> KV append/evict -> chunk attention -> output projection (the DiT blocks of
 * the paper's video pipelines, section 4.2, are where the chunk attention runs).
 *   x      [Nq, d] bf16, the chunk's hidden states (d = heads * head_dim);
 *   w_qkv  [3d, d] bf16, row-major (output features x input features): rows
 *          [0, d) produce q, [d, 2d) k, [2d, 3d) v, each token-major
 *          [Nq, heads, head_dim];
 *   w_o    [d, d] bf16, same convention;
 *   q_buf  [Nq, d] bf16 caller-owned work buffer: receives the rotated q;
 *   o_buf  [Nq, d] bf16 caller-owned work buffer: receives the attention output;
 *   y      [Nq, d] in the stream's out dtype (fp32 or bf16): o_buf . w_o^T.
 * Three launches on the stream's CUDA stream: the QKV projection (its epilogue
 * rounds q/k/v to bf16, rotates q and k, writes q to q_buf and k, v straight
 * into ring slot c mod W), the attention (bf16 output into o_buf), the output
 * projection. Projections accumulate in fp32 on the tensor cores. The chunk
 * counter advances as for frt_kv_append_evict; slot_out / evicted_out (may be
 * NULL) as there. Requires d % 128 == 0. Allowed at the start of a chunk. */
frt_status frt_block_step(frt_stream_t* s, const void* x, const void* w_qkv,
                          const void* w_o, void* q_buf, void* o_buf, void* y,
                          int* slot_out, long long* evicted_out);

/* Plain projection C = A . B^T on the tensor cores (the kernel the block step
 * uses, without its QKV epilogue): A [M, K] bf16 row-major, B [N, K] bf16
 * row-major, C [M, ldc] row-major fp32 (c_dtype FRT_OUT_F32) or bf16
 * (FRT_OUT_BF16), rows/columns past M/N untouched; fp32 accumulation, bf16
 * output rounded to nearest even. K % 8 == 0, ldc >= N, ldc * element size a
 * multiple of 16 bytes, pointers 16-byte aligned. `status` (may be NULL) is a
 * device-visible int[4] that a device-side bounded wait that gave up fills with
 * FRT_ERR_TIMEOUT (it must start zeroed). Enqueued on cuda_stream
 * (cudaStream_t; NULL = legacy default stream). */
frt_status frt_gemm_bf16(const void* a, const void* b, void* c, int M, int N,
                         int K, int ldc, int c_dtype, void* status,
                         void* cuda_stream);
/* Tile plan of the projection kernel for C [M, N] (for reports; no counterpart in the
 * paper): *bn = output columns per tile (128 or 256), *ctas = CTAs per tile (2: a CTA
 * pair on 256 rows, 1: one CTA on 128 rows). qkv = 1 asks for the QKV epilogue of
 * frt_block_step with d = heads * head_dim (N = 3 d). FRT_ERR_INVALID_ARG on NULL
 * outputs or non-positive sizes. Host-only: it launches nothing and reads only the
 * current device's SM count (148 assumed when no device is visible). */
frt_status frt_gemm_plan(int M, int N, int qkv, int d, int* bn, int* ctas);

/* Work split of one chunk-attention launch (for reports and tests; no counterpart in
 * the paper). A launch runs one CTA per work item; a query group is (stream, head, 256
 * query rows). For n streams in launch order with n_q[i] queries and n_kv[i] valid
 * keys, all with `heads` heads, on `sms` SMs (<= 0: the current device's SM count, 148
 * when none is visible): query groups [0, *n_full) run whole and each later group's KV
 * range is cut into *n_split parts whose partials are merged (the plan whose simulated
 * schedule of the launch ends first). FRT_ERR_INVALID_ARG on NULL pointers or sizes
 * < 1. Host-only: it launches nothing. */
frt_status frt_attention_plan(int n, const int* n_q, const long long* n_kv, int heads, int sms,
                              int* n_full, int* n_split);

/* ---- Streaming causal 3D convolution (the VAE-decoder stage) --------------------
 * The paper's video pipelines end in a streaming VAE decoder (Appendix A.3, the
 * DiT -> VAE template: the decoder carries state from one batch to the next, the
 * (V, V, 1) self-edge). Its building block is a causal 3D convolution over a chunk
 * of F frames whose kt - 1 temporal taps reach into a cache of the previous chunk's
 * last frames (zeros before the first chunk). For output frame t, pixel (h, w),
 * channel o:
 *   y = bias[o] + sum over taps (dt, dh, dw), channels c of
 *       w[(dt*kh + dh)*kw + dw][o][c] * x_ext[t + dt][h + dh - kh/2][w + dw - kw/2][c]
 * with x_ext = (cache frames, chunk frames) and zeros outside the frame.
 * Tensors are channels-last: x [F, H, W, Cin] bf16, w [kt*kh*kw, Cout, Cin] bf16,
 * bias [Cout] fp32, y [F, H, W, Cout] fp32 or bf16; device pointers, 16-byte
 * aligned, owned by the caller. A handle owns its frame cache (two [kt-1, H, W, Cin]
 * bf16 buffers used in turn), allocated in frt_conv_configure. Cin and Cout are
 * multiples of 64; 1 <= kt <= 4; kh, kw odd and <= 7. Not thread-safe per handle. */
typedef struct frt_conv frt_conv_t;
/* NULL on invalid sizes (frt_last_error()). */
frt_conv_t* frt_conv_create(int cin, int cout, int kt, int kh, int kw, int grid_h,
                            int grid_w, int frames_per_chunk);
/* Allocate the cache (zeroed) and the status word; set the output dtype and the
 * cudaStream_t every later call enqueues on. May be called again to change them. */
frt_status frt_conv_configure(frt_conv_t* c, int out_dtype, void* cuda_stream);
/* One chunk: y from (cache, x), then the cache becomes the last kt - 1 frames of
 * (cache, x). One launch (the convolution on the tensor cores; its epilogue warps write
 * the next cache into the other half of a ping-pong pair while the MMAs run). */
frt_status frt_conv_step(frt_conv_t* c, const void* x, const void* w,
                         const void* bias, void* y);
/* Tile of the convolution kernel, for tuning and tests (no counterpart in the paper):
 * bn = output channels per tile (64, 96, 128, 192 or 256, dividing Cout) and pair = 1
 * for CTA pairs (tcgen05 cta_group::2, two pixel tiles per pair) or 0 for single
 * CTAs; bn = 0 restores the automatic choice (a cost model of the launch). Applies
 * to later frt_conv_step calls, which return FRT_ERR_UNSUPPORTED for bn = 96 with a
 * bf16 output (staged in 64-channel units). With whole tiles (frt_conv_set_split
 * mode 1) results do not depend on the tile: each output sums its products in one
 * order (temporal tap, channel block, spatial tap). FRT_ERR_INVALID_ARG for other
 * values; may allocate the split workspace (FRT_ERR_OOM). */
frt_status frt_conv_set_tile(frt_conv_t* c, int bn, int pair);
/* Work split of the convolution kernel, for tuning and tests (no counterpart in the
 * paper). The K loop of an output tile is its halos (temporal tap x 64-channel
 * block); the launch's units (CTAs, or CTA pairs) either take whole tiles or, split,
 * equal shares of all tiles' halo steps in order, so that a tile's K sum may come in
 * parts from consecutive units: each part is written to a workspace and the part that
 * arrives last adds them in step order, then the bias. mode 0 = automatic (split
 * when the tiles do not fill the units evenly and the cost model favours it), 1 =
 * whole tiles only, 2 = split whenever the units do not divide the tiles; units = 0
 * for every SM (or SM pair), else at most that many units. Results are deterministic
 * for a given plan; split and whole-tile plans may differ in the last bits (another
 * fp32 summation grouping, within the same error bound). Applies to later
 * frt_conv_step calls; may allocate the workspace (FRT_ERR_OOM). FRT_ERR_INVALID_ARG
 * for a mode outside 0..2 or units < 0. */
frt_status frt_conv_set_split(frt_conv_t* c, int mode, int units);
/* The launch plan frt_conv_step would use for these sizes on a GPU with `sms` SMs
 * (host-only, launches nothing): bn and pair as frt_conv_set_tile (0 = automatic),
 * split_mode and units as frt_conv_set_split. Writes plan[0..5] = tile width, pair
 * (0/1), units (CTAs or CTA pairs in the grid), split (0/1), number of output tiles
 * (pair tiles count once), halos per tile (the K steps: kt x Cin / 64).
 * FRT_ERR_INVALID_ARG on invalid sizes, FRT_ERR_UNSUPPORTED if no tile fits. */
frt_status frt_conv_plan(int cin, int cout, int kt, int kh, int kw, int grid_h, int grid_w,
                         int frames_per_chunk, int out_dtype, int sms, int bn, int pair,
                         int split_mode, int units, int* plan);
/* The current cache [kt-1, H, W, Cin] bf16 (device, read-only use). */
frt_status frt_conv_cache(const frt_conv_t* c, const void** cache);
/* Wait for the handle's work; returns FRT_ERR_TIMEOUT if a device wait gave up. */
frt_status frt_conv_sync(frt_conv_t* c);
/* Zero the cache and the status word (synchronises first). */
frt_status frt_conv_reset(frt_conv_t* c);
void frt_conv_destroy(frt_conv_t* c);

/* Operation 3 for n independent streams in one launch (ragged KV lengths; streams hold
 * disjoint persistent state, so they carry no cross-stream edge: section 3.2 "IR
 * design", node-level state annotation):
 * each streams[i] must have just appended (as for frt_chunk_attention); q[i]
 * and out[i] are that stream's rotated queries and output. All streams must
 * share heads, head_dim, sm_scale and out dtype; work is ordered longest KV
 * first and enqueued on streams[0]'s CUDA stream, which first waits for the
 * other streams' CUDA streams (events), and which they wait for afterwards.
 * 1 <= n <= 32, no stream repeated. */
frt_status frt_chunk_attention_batched(frt_stream_t* const* streams, int n,
                                       const void* const* q, void* const* out);

/* Operation 3 for callers that cannot allocate device memory (no counterpart in
 * the paper). Some callers may not call cudaMalloc: code under a memory planner or
 * arena that owns every device byte, real-time loops where an allocation (which can
 * synchronise the device) is not allowed, integrations whose only device memory is
 * what they pass in. This call allocates nothing: no stream handle, no cudaMalloc,
 * cudaFree or allocating library routine. It computes the same attention as
 * frt_chunk_attention, out[i,h,:] = sum_j softmax_j(scale <q[i,h], k[j,h]>) v[j,h,:]
 * over all n_kv rows of caller-owned buffers:
 *   q    device [n_q, heads, head_dim] bf16 (already rotated);
 *   k, v device [n_kv, heads, head_dim] bf16 (e.g. the valid prefix of a cache);
 *   out  device [n_q, heads, head_dim], fp32 or bf16 (out_dtype);
 *   sm_scale <= 0 selects 1/sqrt(head_dim);
 *   status optional device pointer to 4 ints, zeroed by the caller, where a device
 *        bounded-wait timeout records FRT_ERR_TIMEOUT (NULL: not recorded);
 *   cuda_stream the cudaStream_t the work is enqueued on (NULL = legacy stream).
 * All pointers 16-byte aligned; head_dim 64 or 128. The kernel's split-KV scratch
 * lives in one static device array of this library (8 MiB of partials, 4096 merge
 * counters) that every GPU loading the library holds until exit; splits are limited
 * to what it holds, and heads * ceil(n_q / 256) > 4096 is rejected with
 * FRT_ERR_UNSUPPORTED. The first call in each CUDA context (the device's primary
 * context, another context the caller made current, or a new primary context after
 * cudaDeviceReset) looks up the array's device address in that context; make that
 * first call before any stream capture. All calls share the
 * array and each clears its merge counters on the stream first: calls that overlap
 * on the GPU (other streams, other threads) race and must not be issued.
 * frt_last_error() describes an error this call returns. */
frt_status frt_chunk_attention_noalloc(const void* q, const void* k, const void* v,
                                       void* out, int n_q, int n_kv, int heads,
                                       int head_dim, double sm_scale, int out_dtype,
                                       void* status, void* cuda_stream);

/* Per-denoising-step caches. Each denoising step of the DiT keeps its own KV cache
 * (section 3.1 "Case study"; Appendix A.4: step Q_i of batch j+1 depends only on
 * step Q_i of batch j), which is what makes pipelining across steps legal. A step
 * group owns n_steps independent streams of one shape; frt_steps_tick advances the
 * active steps of one pipeline tick: in the wavefront schedule step i works on chunk
 * t - i at tick t, so the steps' attentions are independent and run as ONE batched
 * launch (the single-GPU form of the paper's stage pipeline over denoising steps).
 * 1 <= n_steps <= 32; all steps share one frt_config (and CUDA stream). */
typedef struct frt_steps frt_steps_t;
frt_steps_t* frt_steps_create(int n_steps, int heads, int head_dim, int tokens_per_frame,
                              int frames_per_chunk, int window_chunks);
frt_status frt_steps_configure(frt_steps_t* g, const frt_config* cfg);
/* The stream of step `step` (owned by the group; do not destroy it). NULL if out of range. */
frt_stream_t* frt_steps_stream(const frt_steps_t* g, int step);
/* One tick: for every step i with bit i of active_mask set, rotate q[i], k[i] in place
 * (frt_rope3d_qk at that step's own chunk counter), append (k[i], v[i]) to its cache,
 * then one batched attention launch writes out[i] for all active steps. Arrays are
 * indexed by step; entries of inactive steps are ignored. */
frt_status frt_steps_tick(frt_steps_t* g, unsigned int active_mask, void* const* q,
                          void* const* k, const void* const* v, void* const* out);
void frt_steps_destroy(frt_steps_t* g);

/* Wait for the stream's work and return its device status (no counterpart in the
 * paper; the library's error channel) (FRT_OK or the
 * first device error, e.g. FRT_ERR_TIMEOUT). */
frt_status frt_stream_sync(frt_stream_t* s);

/* Start the stream over, as a new video would (the state edge of section 2 has no
 * predecessor for batch 0): clear the cache contents, chunk counter, ordering state, split-KV merge
 * counters and device status (the way back after FRT_ERR_TIMEOUT). */
frt_status frt_stream_reset(frt_stream_t* s);

/* Release everything the handle owns (waits for its work first). NULL is a no-op. */
void frt_stream_destroy(frt_stream_t* s);

/* Snapshot of the stream's persistent state (the paper's cross-batch state edge, section
 * 2; moving it between resources is the kappa cost of Appendix A.1.2): enqueue copies of
 * the whole ring (K and V, rows = window_chunks * Nq each, [rows, heads, head_dim] bf16)
 * into k_dst / v_dst (device or pinned host memory, caller-owned) on the stream's CUDA
 * stream, and report the chunk counter. The copies are complete when frt_stream_sync
 * returns. Not allowed between frt_rope3d_qk and the append (FRT_ERR_STATE). */
frt_status frt_stream_save(frt_stream_t* s, void* k_dst, void* v_dst, long long* counter);

/* Load a snapshot taken by frt_stream_save (from this stream or another of the same
 * shape) and continue from it: the ring is overwritten from k_src / v_src (enqueued on
 * the stream), the counter set, and the next call must start a chunk. The chunks that
 * follow produce the outputs the saved stream would have produced, bit for bit. */
frt_status frt_stream_restore(frt_stream_t* s, const void* k_src, const void* v_src,
                              long long counter);

/* Race and overrun detection (no counterpart in the paper). Every ring buffer sits
 * between guard words written at configure; this call waits for the stream's work and
 * compares them: FRT_ERR_BOUNDS (naming the guard) if a kernel wrote past either end of
 * the K or V ring, else FRT_OK. The FRT_DEBUG build of the library also runs it inside
 * every frt_stream_sync, and its kernels check every derived index (work items, ring
 * rows, split-KV rows) against the launch's extents: an access outside is skipped and
 * FRT_ERR_BOUNDS recorded in the stream's status (no trap). */
frt_status frt_stream_check_guards(frt_stream_t* s);

/* 1 if this library was built with FRT_DEBUG (bounds-checking kernels), else 0. */
int frt_debug_build(void);

/* Read-only view of the stream's ring buffer for inspection and snapshots: device
 * pointers of the K and V caches ([rows, heads, head_dim] bf16, rows = W * Nq; chunk c
 * occupies rows [(c mod W) * Nq, (c mod W + 1) * Nq)). Valid until destroy. */
frt_status frt_stream_cache(const frt_stream_t* s, const void** k_cache,
                            const void** v_cache, long long* rows);

/* Instrumentation: record start_event / stop_event (cudaEvent_t, created by the
 * caller) on the stream's CUDA stream immediately before and after every
 * attention kernel launch of s (frt_chunk_attention, frt_chunk_step and batched
 * launches led by s) until called again; NULL, NULL turns it off. */
frt_status frt_stream_set_attention_events(frt_stream_t* s, void* start_event,
                                           void* stop_event);

/* Instrumentation: the same for every KV append kernel launch of s
 * (frt_kv_append_evict and the append inside frt_chunk_step). */
frt_status frt_stream_set_append_events(frt_stream_t* s, void* start_event, void* stop_event);

/* Instrumentation for frt_block_step: events recorded immediately before and
 * after its QKV projection (qkv_*) and its output projection (out_*) launches;
 * the attention launch uses the attention events. NULLs turn it off. */
frt_status frt_stream_set_block_events(frt_stream_t* s, void* qkv_start,
                                       void* qkv_stop, void* out_start,
                                       void* out_stop);

/* Index of the next chunk to be appended (chunks appended so far). */
long long frt_stream_chunk_counter(const frt_stream_t* s);

/* Host-only sliding-window arithmetic used by frt_kv_append_evict: for chunk
 * index `chunk` >= 0 and window >= 1, the ring slot (chunk mod window), the
 * evicted chunk (chunk - window, or -1) and the valid chunk count after the
 * append (min(chunk + 1, window)). Any output pointer may be NULL. */
frt_status frt_window_index(long long chunk, int window, int* slot,
                            long long* evicted, int* valid_chunks);

const char* frt_status_string(frt_status st);

/* Thread-local description of the last error returned on this thread. */
const char* frt_last_error(void);

/* Library version string. */
const char* frt_version(void);

#ifdef __cplusplus
}
#endif
#endif /* FRT_H */
