/*
 * hs_debug.h - test hooks into libhs's tensor-core kernels.
 *
 * Not part of the training API.  hs_debug_gemm_bf16 runs one product through
 * the same tcgen05/TMA kernel that hs_step uses for the per-worker forward and
 * backward passes (Eq. 1's per-worker gradients g^m, Section 1);
 * hs_debug_wgrad_avg runs the kernel that forms the per-worker weight gradients
 * of a layer, averages them and applies the update.  Tests check each kernel in
 * isolation against a plain reference.  All matrix pointers are device
 * pointers, row-major, with leading dimensions in elements; the calls are
 * synchronous (they wait for the kernel and report launch/runtime errors).
 */
#ifndef HS_DEBUG_H_
#define HS_DEBUG_H_

#include <stdint.h>

#include "hs.h"

#ifdef __cplusplus
extern "C" {
#endif

enum {
  HS_GEMM_FWD_RELU = 0,   /* D bf16 [M,N] = relu(A[M,K] B[N,K]^T + bias[N])           */
  HS_GEMM_FWD_LOGITS = 1, /* D fp32 [M,N] = A[M,K] B[N,K]^T + bias[N]                  */
  HS_GEMM_DGRAD = 2,      /* D bf16 [M,N] = (A[M,K] B[K,N]) * (Z[M,N] > 0)              */
  HS_GEMM_WGRAD = 3       /* D_g fp32 [M,N] = A[k_g, M]^T B[k_g, N] for each group g:   */
                          /*   rows k of A [K,M] and B [K,N] in [k_off[g], k_off[g+1]), */
                          /*   D_g at D + g * d_gstride                                  */
};

/* Kernel form, OR-ed into mode: 0 = the library's current form, HS_GEMM_FORM_SINGLE = one SM per
 * 128 x 256 tile, HS_GEMM_FORM_PAIR = a two-SM cluster per 256 x 256 tile (tcgen05 cta_group::2). */
enum { HS_GEMM_FORM_SINGLE = 0x100, HS_GEMM_FORM_PAIR = 0x200 };

/* OR-ed into mode: the kernel's TMA producer issues no loads, so the MMA issuer's bounded wait on
 * the first stage expires (2 s of %globaltimer) and the kernel leaves through its error path:
 * status word set, abort flag raised for the other roles, tensor memory freed, no fault.  The
 * call then returns HS_ERR_DEVICE_CHECK.  Exercises the device-side failure detection. */
enum { HS_GEMM_TEST_STALL = 0x1000 };

/* A, B, Z: bf16; bias: fp32 [N]; k_offsets_host: host int32 [groups+1] (HS_GEMM_WGRAD only,
 * else NULL with groups = 1).  Returns HS_ERR_INVALID_ARG for shapes the kernel cannot take
 * (leading dimensions must be multiples of 8 elements, pointers 16-byte aligned),
 * HS_ERR_CUDA on a launch or runtime error, HS_ERR_DEVICE_CHECK when a bounded wait in the
 * kernel expired. */
hs_status hs_debug_gemm_bf16(int32_t mode, int32_t M, int32_t N, int32_t K, const void* A, int64_t lda,
                             const void* B, int64_t ldb, void* D, int64_t ldd, const float* bias,
                             const void* Z, int64_t ldz, const int32_t* k_offsets_host, int32_t groups,
                             int64_t d_gstride, void* stream);

/* The per-worker weight gradients of one layer averaged in tensor memory with the update fused
 * (the kernel hs_step uses for large bf16 MLP layers; Eq. 1's g^m, the weighted average of
 * Section 1 / Section 4.2, theta <- theta - lr * g), run alone:
 *   theta[M, N] <- theta - lr * sum_g wavg[g] * A[k_g, M]^T B[k_g, N]   (g = 0 .. groups-1 in order)
 *   shadow[M, N] = bf16(new theta)
 * with rows k_g = [k_offsets_host[g], k_offsets_host[g+1]) of A (bf16 [K][M], MN-major, leading
 * dimension lda) and B (bf16 [K][N], ldb).  theta: device fp32, leading dimension ld_theta,
 * updated in place; shadow: device bf16, ld_shadow; wavg: device fp32 [groups].  groups in
 * 1..32, every group at least one row; leading dimensions multiples of 8 elements, pointers
 * 16-byte aligned.  test_stall = 1: the kernel's loads are never issued, its bounded waits expire
 * (2 s) and the call returns HS_ERR_DEVICE_CHECK with theta unchanged (the failure-detection
 * test).  Synchronous; HS_ERR_INVALID_ARG / HS_ERR_CUDA / HS_ERR_DEVICE_CHECK as above. */
hs_status hs_debug_wgrad_avg(int32_t M, int32_t N, const void* A, int64_t lda, const void* B, int64_t ldb,
                             const int32_t* k_offsets_host, int32_t groups, const float* wavg, float lr,
                             float* theta, int64_t ld_theta, void* shadow, int64_t ld_shadow, int32_t test_stall,
                             void* stream);

#ifdef __cplusplus
}
#endif

#endif /* HS_DEBUG_H_ */
