/*
 * psppo_diag.h -- diagnostic entry points of libpsppo.
 *
 * The paper has no counterpart for these: they expose, for tests, the two pieces
 * of machinery that the update pass is built on. Conventions (device pointers,
 * workspace status word, stream ordering, ps_status returns) are those of psppo.h.
 */
#ifndef PSPPO_DIAG_H_
#define PSPPO_DIAG_H_

#include "psppo.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * The tensor-core contraction under the forward and backward: C[M][N] (+)= A B with
 * bf16 operands and f32 accumulation (tcgen05, TMEM accumulators, TMA-fed).
 * A(m, k) is A[m*lda + k] (a_mn_major = 0, K-major) or A[k*lda + m] (a_mn_major = 1);
 * B(k, n) is B[n*ldb + k] (b_mn_major = 0, K-major) or B[k*ldb + n] (b_mn_major = 1).
 * C is f32 [M][ldc], overwritten (accumulate = 0) or added to (accumulate = 1).
 * variant selects the kernel: 0 = one CTA per 128 x 256 tile (the forward and the logit
 * recompute), 1 = two CTAs of a cluster per 256 x 256 tile (tcgen05 cta_group::2), 2 = one
 * CTA per 256 x 256 tile as two M = 128 halves sharing B (dH and dW).
 * lda, ldb multiples of 8; ldc a multiple of 4; 16-byte aligned A, B, C.
 * ws: at least 256 bytes. sm_103 only (PS_ERR_UNSUPPORTED elsewhere).
 */
int ps_diag_gemm_bf16(int M, int N, int K, int a_mn_major, int b_mn_major, const void* A, int64_t lda,
                      const void* B, int64_t ldb, float* C, int64_t ldc, int accumulate, int variant,
                      void* ws, size_t ws_bytes, ps_stream_t stream);

/*
 * Launch one CTA that waits on a shared-memory barrier that nothing ever completes,
 * using the same bounded wait as the GEMM pipeline. After about timeout_ns
 * (<= 10 s) the wait gives up and sets PS_DEV_TIMEOUT in the workspace status word;
 * ps_workspace_status() then returns PS_ERR_TIMEOUT and the context stays usable.
 */
int ps_diag_wait_timeout(uint64_t timeout_ns, void* ws, size_t ws_bytes, ps_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* PSPPO_DIAG_H_ */
