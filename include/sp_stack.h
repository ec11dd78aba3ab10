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

/* Stack glue (the linear-only stack of the Sec. 3.4 decode measurements, defined above; the
 * paper defines no such glue): out[m, j] = in[m, col0 + j] for m < M, j < ncols; in has row
 * stride in_stride elements.
 * ncols, col0 and in_stride must be multiples of 8. */
sp_status sp_copy_columns(void* out, const void* in, int64_t M, int64_t in_stride, int64_t col0, int64_t ncols,
                          void* stream);

/* Stack glue (as above): h[m, j] = bf16(h[m, j] + a[m, j] + r[j]) in place; h, a [M, N], r [N];
 * N % 8 == 0. */
sp_status sp_residual_add(void* h, const void* a, const void* r, int64_t M, int64_t N, void* stream);

/* Stack glue (as above; the gate * up product of a Llama MLP): out[m, j] = bf16(g[m, j] *
 * g[m, F + j]) for j < F; g [M, 2F], out [M, F]; F % 8 == 0. */
sp_status sp_mul_halves(void* out, const void* g, int64_t M, int64_t F, void* stream);

/* Stack glue, the same product for a gate/up weight whose rows are interleaved (gate_j,
 * up_j): out[m, j] = bf16(g[m, 2j] * g[m, 2j + 1]) for j < F; g [M, 2F], out [M, F];
 * F % 8 == 0.  (Library plumbing: the tensor-core path's counterpart of the pair-product
 * epilogue of sp_linear_epi below.) */
sp_status sp_mul_pairs(void* out, const void* g, int64_t M, int64_t F, void* stream);


/* ---------------------------------------------------------------- chained decode step
 * A chain of sparse linears run by one persistent launch (a decode step through the
 * layers of a model).  Linear k computes acc = x_k . (W_k o Mask_k)^T (FP32 accumulation;
 * Sec. 2.4.2's compressed submatrices streamed from global memory and expanded on chip)
 * and writes it through one of the epilogues below.  Every linear waits for the previous
 * one to be complete (its x may be any earlier output), while the compressed weights of
 * all linears stream from HBM without a break between linears.  Results equal those of
 * the corresponding sp_linear calls and sp_stack glue up to FP32 summation order, and are
 * bitwise repeatable for a given (chain, m, device). */
typedef enum sp_chain_epilogue {
  SP_EPI_STORE = 0,        /* y[m, n] = bf16(acc)                                          */
  SP_EPI_RESIDUAL = 1,     /* y[m, n] = bf16((y[m, n] + bf16(acc)) + r[n]), in place      */
  SP_EPI_PAIR_PRODUCT = 2  /* rows 2j and 2j+1 (N even): y[m, j] = bf16(bf16(acc_2j) *
                              bf16(acc_2j+1)) -- the gate*up product when the rows of the
                              fused gate/up weight are interleaved (gate_j, up_j)          */
} sp_chain_epilogue;

typedef struct sp_chain_op {
  const sp_matrix* w;  /* compressed weight [N, K] (INT8: bf16(acc) is bf16(s[n] * acc))   */
  const void* x;       /* bf16 input [m, K] with row stride ldx elements (ldx >= K)        */
  int64_t ldx;
  void* y;             /* bf16 output, row stride ldy (>= N, or >= N/2 for the pair product) */
  int64_t ldy;
  const void* r;       /* bf16 [N] residual vector for SP_EPI_RESIDUAL, else NULL           */
  int32_t epilogue;    /* sp_chain_epilogue */
  int32_t reserved;    /* 0 */
} sp_chain_op;

/* Workspace bytes that sp_chain_run needs on the current device (0 for m == 0); library
 * plumbing with no counterpart in the paper. */
sp_status sp_chain_workspace_size(int64_t m, size_t* bytes);

/* The chained decode step described above (each op a Sec. 2.4.2 sparse linear with its
 * epilogue).  Run ops[0], ops[1], ..., ops[n_ops - 1] in order for m batch rows (1 <= m <= 4;
 * SP_ERR_UNSUPPORTED above).  All weights live on the current device and hold the same
 * value type (bf16 or INT8).  x, y and r are 2-byte aligned (any row stride); the workspace
 * is 16-byte aligned.  The workspace (sp_chain_workspace_size bytes) is zero-filled before
 * its first use, and every call leaves it ready for the next; calls that share it must be
 * ordered on one stream.  After SP_ERR_TIMEOUT from sp_check, zero it again.  Each group
 * of up to 160 linears is one launch (all its CTAs resident at once, launched
 * cooperatively); the launch allocates nothing and does not synchronise the host.
 * m == 0 or n_ops == 0 returns SP_OK without a launch. */
sp_status sp_chain_run(const sp_chain_op* ops, int32_t n_ops, int64_t m, void* workspace_dev, size_t workspace_bytes,
                       void* stream);

/* One sparse linear (Sec. 2.4.2) with the stack's glue folded into its output: y =
 * epilogue(x . (W o Mask)^T) with the epilogues of sp_chain_epilogue -- SP_EPI_STORE as
 * sp_linear; SP_EPI_RESIDUAL y[m, n] = bf16((y[m, n] + bf16(acc)) + r[n]) in place;
 * SP_EPI_PAIR_PRODUCT y[m, j] = bf16(bf16(acc_2j) * bf16(acc_2j+1)), y [m, N/2] (N even).
 * The epilogue's results equal those of sp_linear followed by sp_residual_add or
 * sp_mul_pairs (bitwise, for the same kernel and batch).  x [m, K] and y are bf16,
 * contiguous and 16-byte aligned; r is bf16 [N] for SP_EPI_RESIDUAL, else NULL; the
 * workspace is as for sp_linear (sp_workspace_size bytes, zero-filled once, calls that
 * share it ordered on one stream).  Runs on the CUDA-core kernels: where the automatic path
 * takes the tensor-core kernel for m rows the call returns SP_ERR_UNSUPPORTED without a
 * launch, and the caller uses sp_linear and the glue call instead.  Other errors as
 * sp_linear, and SP_ERR_INVALID_ARG for an unknown epilogue, a missing r or an odd N with
 * the pair product. */
sp_status sp_linear_epi(const sp_matrix* h, const void* x, int64_t m, void* y, int32_t epilogue, const void* r,
                        void* workspace_dev, size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SP_STACK_H */
