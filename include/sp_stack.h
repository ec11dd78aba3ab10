/*
 * sp_stack.h -- elementwise glue for chaining sparse linears into a decode step of a
 * Llama-2-7B linear stack (libsp, GB300 / sm_103a).
 *
 * The paper has no definition of a linear-only stack: its deployment measurements run
 * whole Llama-2-7B models (Sec. 3.4).  The benchmark stack keeps only the seven linear
 * layers per block (as four fused launches: qkv, o, gate/up, down), with no attention or
 * normalisation, and chains them with residual adds:
 *     v  = qkv(h)[:, 2*D : 3*D]                 (sp_copy_columns; D = 4096)
 *     h  = h + o(v) + r                          (sp_residual_add)
 *     a  = gu(h)[:, :F] * gu(h)[:, F:]           (sp_mul_halves; F = 11008)
 *     h  = h + down(a) + r'                      (sp_residual_add)
 * with r, r' fixed bf16 vectors per layer.  All tensors are bf16, row-major, 16-byte
 * aligned device memory; arithmetic is FP32 with one bf16 round-to-nearest-even per
 * output.  Every call is asynchronous on `stream` (a cudaStream_t as void*) and returns
 * an sp_status; none allocates.
 */
#ifndef SP_STACK_H
#define SP_STACK_H

#include <stdint.h>

#include "sp.h"

#ifdef __cplusplus
extern "C" {
#endif

/* out[m, j] = in[m, col0 + j] for m < M, j < ncols; in has row stride in_stride elements.
 * ncols, col0 and in_stride must be multiples of 8. */
sp_status sp_copy_columns(void* out, const void* in, int64_t M, int64_t in_stride, int64_t col0, int64_t ncols,
                          void* stream);

/* h[m, j] = bf16(h[m, j] + a[m, j] + r[j]) in place; h, a [M, N], r [N]; N % 8 == 0. */
sp_status sp_residual_add(void* h, const void* a, const void* r, int64_t M, int64_t N, void* stream);

/* out[m, j] = bf16(g[m, j] * g[m, F + j]) for j < F; g [M, 2F], out [M, F]; F % 8 == 0. */
sp_status sp_mul_halves(void* out, const void* g, int64_t M, int64_t F, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SP_STACK_H */
