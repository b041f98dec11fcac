/* Dense matrix product (fp32 activations, bf16 weights) of the prompt prefill, exposed on its own
 * (sm_103a).
 *
 * A prefill pass computes, for every token of a prompt, the products of the stage's weight
 * matrices with that token's activations (section III: a stage applies its blocks to each token;
 * the prefill phase of time to first token, section VI, instrumentation paragraph).  With the
 * tokens as rows this is Y = X W^T, run on the tensor cores (tcgen05.mma, fp32 accumulation in
 * tensor memory, operands staged by TMA).  kfl_stage_prefill calls the same kernel with fused
 * epilogues; this entry point returns the plain product so that it can be checked on its own.
 *
 * Conventions as in kafila_stage.h.
 */
#ifndef KAFILA_GEMM_H
#define KAFILA_GEMM_H

#include <stdint.h>

#include "kafila_stage.h"

#ifdef __cplusplus
extern "C" {
#endif

/* y[t][n] = sum_k x[t][k] w[n][k] for t < T, n < N, in fp32.  x is split into two bf16 terms
 * (hi = bf16(x), lo = bf16(x - hi)) that both meet each bf16 weight on the tensor cores, so the
 * result is that of fp32 x up to about 2^-16 relative, with fp32 sums (their order is the
 * kernel's).
 *   x  device fp32 [T][ldx], ldx >= K
 *   w  device bf16 [N][K] row-major (the nn.Linear convention); read only
 *   y  device fp32 [T][ldy], ldy >= N and a multiple of 4, 16-byte aligned; columns >= N untouched
 * The weights are copied into the decode path's tile layout and x into its two terms (one
 * temporary device buffer) first.  Synchronous on cuda_stream.  Errors: KFL_ERR_ARG (sizes,
 * strides, alignment, NULL pointers), KFL_ERR_OOM, KFL_ERR_CUDA, KFL_ERR_TIMEOUT (a bounded wait
 * of the kernel's pipeline gave up). */
int kfl_matmul_bf16w(const float *x, int T, int K, int ldx, const uint16_t *w, int N, float *y, int ldy,
                     void *cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* KAFILA_GEMM_H */
