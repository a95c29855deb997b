/*
 * frt_selftest.h — self-test entry points of libfrt.so, used by the GPU tests to
 * check the hardware building blocks of the attention kernel in isolation. They are
 * not part of the streaming API (include/frt.h) and have no counterpart in the paper.
 */
#ifndef FRT_SELFTEST_H
#define FRT_SELFTEST_H
#include "frt.h"
#ifdef __cplusplus
extern "C" {
#endif

/* One 128x128x128 bf16 tile, C = A * op(B), fp32, through TMA (128-byte swizzle) into
 * shared memory, tcgen05.mma into TMEM and tcgen05.ld back to registers.
 *   a: device [128, 128] bf16 row-major (row m, reduction index k contiguous).
 *   b: device [128, 128] bf16 row-major; b_mn_major = 0: b[n][k] (C = A B^T, the QK^T
 *      layout); b_mn_major = 1: b[k][n] (C = A B, the PV layout).
 *   lbo_b, sbo_b: descriptor byte offsets for the MN-major B (16 <= x <= 16384).
 *   a_from_tmem: 1 stages A in TMEM (packed bf16 pairs) and uses the A-from-TMEM MMA.
 *   c: device [128, 128] fp32 row-major; dev_status: device int set to 1 on a timeout.
 * Enqueued on cuda_stream; returns 0 on launch success, < 0 on an argument/launch error. */
int frt_selftest_umma_tile(const void* a, const void* b, float* c, int b_mn_major, int lbo_b,
                           int sbo_b, int a_from_tmem, int* dev_status, void* cuda_stream);

/* A CTA pair (cluster of 2) computes one 256x128x128 bf16 tile C = A B^T with
 * tcgen05.mma.cta_group::2: CTA r loads rows [128r, 128r+128) of A and rows
 * [64r, 64r+64) of B with TMA (completion signalled on the leader CTA's mbarrier),
 * the leader issues the MMAs, each CTA reads its 128 rows of D from its TMEM.
 *   a: device [256, 128] bf16 row-major; b: device [128, 128] bf16 row-major (b[n][k]);
 *   c: device [256, 128] fp32; taddrs: device uint32[2], the TMEM address each CTA got
 *   from the pair allocation; dev_status: device int set to 1 on a timeout.
 * Returns 0 on launch success, < 0 on an argument/launch error. */
int frt_selftest_umma_pair(const void* a, const void* b, float* c, unsigned* taddrs,
                           int* dev_status, void* cuda_stream);

/* The P.V form of the same pair MMA: A (device [256, 128] bf16, row-major) is staged in
 * TMEM (CTA r its rows [128 r, 128 r + 128), packed bf16 pairs) and used as the TMEM
 * operand; b is device [128, 128] bf16 row-major read as the MN-major B (K rows x N
 * columns), CTA r holding N columns [64 r, 64 r + 64). c = A . b, device [256, 128] fp32.
 * Returns 0 on launch success, < 0 on an argument/launch error. */
int frt_selftest_umma_pair_pv(const void* a, const void* b, float* c, unsigned* taddrs,
                              int* dev_status, void* cuda_stream);

/* Force the output-column tile width of every later projection launch (frt_gemm_bf16,
 * frt_block_step, frt_gemm_plan) to bn in {128, 192, 256}; 0 restores the automatic
 * choice. Process-wide and not thread-safe: for tests that cover every width. Returns
 * 0, or -1 for another value. */
int frt_selftest_gemm_force_bn(int bn);

/* How the convolution kernel's split tiles gather their parts in every later
 * frt_conv_step: 0 as built; 1 without the watch while the first part's MMAs run (the
 * other parts come only afterwards, by bulk copies into the idle rings); 2 with neither
 * the watch nor the wait afterwards (the first part writes itself and arrives, and the
 * part that completes the count adds them all). Every mode gives the same result.
 * Process-wide and not thread-safe: for tests that cover each path. Returns 0, or -1
 * for another value. */
int frt_selftest_conv_part_mode(int mode);

/* Launch a kernel whose one waiting thread waits on an mbarrier that nothing arrives
 * on, bounded by limit_ns (<= 100 ms); it must record FRT_ERR_TIMEOUT in s's status
 * block, which frt_stream_sync then returns. s must be configured. */
frt_status frt_selftest_wait_timeout(frt_stream_t* s, long long limit_ns, void* cuda_stream);

/* Debug build only (FRT_DEBUG): the next append of any stream aims its stores one ring
 * slot past the end of the cache. The kernel's bounds check must refuse them and record
 * FRT_ERR_BOUNDS; the debug build keeps one chunk of slack after the rear guard, so the
 * stores would still land in the library's own memory if the check missed them (and the
 * guard check would report it). FRT_ERR_UNSUPPORTED in a release build. */
frt_status frt_selftest_append_past_ring(void);

/* Overwrite one byte of a guard word of s (which: 0 K front, 1 V front, 2 K rear, 3 V
 * rear) from the host, to check that frt_stream_check_guards reports it. */
frt_status frt_selftest_poke_guard(frt_stream_t* s, int which);

#ifdef __cplusplus
}
#endif
#endif
