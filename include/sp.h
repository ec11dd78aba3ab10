/*
 * sp.h -- C ABI of libsp: bitmask-compressed unstructured-sparse linear layers
 * y = x . (W o Mask)^T on one NVIDIA GB300 (sm_103a).
 *
 * Method.  The weight is stored the way the paper's GPU engine stores it
 * (Sec. 2.4.2): cut into submatrices, each kept as its dense nonzero values plus
 * a bitmask; at run time the submatrices are streamed from global memory and
 * expanded on chip by the bitmask (the per-block bitmask encoding itself is the
 * one of Sec. 2.4.1).  Decode-sized batches are bound by reading the compressed
 * bytes; prefill-sized batches run the expanded tiles on the tensor cores.
 *
 * Compressed format (identical bytes on every GPU; see also the constants below).
 *   The matrix [N, K] is cut into T = ceil(K/64) K-tiles and RB = ceil(N/128)
 *   row blocks.  Chunk (rb, t) is number c = rb*T + t and starts at byte off[c]
 *   of the buffer (off[0] = 0, off[RB*T] = total size, all multiples of 16):
 *     bytes [0, 1024)   128 little-endian uint64 masks, one per row 128*rb + r;
 *                       bit j (LSB = 0) set <=> column 64*t + j is kept.
 *                       Rows >= N and columns >= K have no bits.
 *     then              the kept values of row 0, row 1, ..., row 127 of the
 *                       chunk, each row in ascending column order (bf16 bit
 *                       patterns, 2 bytes; or int8, 1 byte), no gaps;
 *     then              zero bytes up to the next multiple of 16.
 *   INT8 matrices also carry one fp32 scale per output row: w[n,k] = q[n,k]*s[n].
 *
 * Conventions for every call.
 *   - Device pointers point to memory of the current CUDA device, row-major and
 *     contiguous, and must be 16-byte aligned (else SP_ERR_ALIGNMENT).
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  Calls are asynchronous on that stream unless stated otherwise;
 *     the caller keeps every buffer alive until the stream has passed the call.
 *   - No call aborts, traps or prints.  Every call returns a status.  Kernel
 *     waits are bounded: a wait that expires records SP_ERR_TIMEOUT in a device
 *     status word that sp_check() reports.
 *   - There is no CPU fallback: without a usable GPU the calls that need one
 *     return SP_ERR_CUDA.
 */
#ifndef SP_H
#define SP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SP_TILE_K 64            /* columns per K-tile (one uint64 mask per row) */
#define SP_CHUNK_ROWS 128       /* rows per chunk */
#define SP_CHUNK_MASK_BYTES 1024
#define SP_CHUNK_ALIGN 16

typedef enum sp_status {
  SP_OK = 0,
  SP_ERR_INVALID_ARG = 1,   /* null pointer, negative or zero size, bad enum */
  SP_ERR_UNSUPPORTED = 2,   /* valid but not supported (e.g. K % 8 != 0) */
  SP_ERR_ALIGNMENT = 3,     /* a pointer is not 16-byte aligned */
  SP_ERR_CUDA = 4,          /* a CUDA runtime call or a launch failed */
  SP_ERR_OUT_OF_MEMORY = 5, /* the allocator returned NULL */
  SP_ERR_TIMEOUT = 6,       /* a bounded device wait expired (reported by sp_check) */
  SP_ERR_BAD_HANDLE = 7,    /* not a live sp_matrix */
  SP_ERR_WORKSPACE = 8      /* workspace missing or smaller than sp_workspace_size() */
} sp_status;

typedef enum sp_dtype { SP_BF16 = 0, SP_INT8 = 1 } sp_dtype;

/* Kernel family used by sp_linear_ex.  SP_PATH_AUTO picks by batch size M: the CUDA-core
   family for M <= 10 (bf16 values) or M <= 13 (int8 values), the tensor-core family above
   (the measured crossover on the Llama-2-7B shapes). */
typedef enum sp_path {
  SP_PATH_AUTO = 0,
  SP_PATH_CUDA_CORE = 1,    /* popc-prefix expansion, FP32 FMA on CUDA cores */
  SP_PATH_TENSOR_CORE = 2   /* expansion into tensor memory, tcgen05 MMA */
} sp_path;

typedef struct sp_matrix sp_matrix; /* opaque; owns the compressed weight */

typedef struct sp_info_t {
  int64_t n, k;             /* logical shape [N, K] */
  int64_t tiles, row_blocks;
  int32_t dtype;            /* sp_dtype */
  int32_t device;           /* CUDA device the buffers live on */
  int64_t nnz;              /* kept entries */
  uint64_t bytes;           /* size of the compressed buffer (padding included) */
  uint64_t max_chunk_bytes; /* largest single chunk */
  uint64_t scale_bytes;     /* 4*N for INT8, else 0 */
} sp_info_t;

/* Device allocator callbacks.  alloc returns a device pointer of at least `bytes`
 * bytes, 256-byte aligned, or NULL; free releases it.  Passing NULL for both uses
 * cudaMalloc / cudaFree.  The library calls them only inside sp_compress,
 * sp_clone and sp_free. */
typedef void* (*sp_alloc_fn)(size_t bytes, void* ctx);
typedef void (*sp_free_fn)(void* ptr, void* ctx);

/* Compress W o Mask (the storage of Sec. 2.4.2).
 *   w_dev      [N, K] bf16 bit patterns (SP_BF16) or int8 values (SP_INT8).
 *   mask_dev   [N, K] uint8, nonzero = kept.  A kept zero is stored as a value;
 *              a masked-out nonzero is dropped.
 *   scale_dev  [N] fp32 per-row scales for SP_INT8 (copied); must be NULL for SP_BF16.
 *   N, K       N >= 1, K >= 1, K % 8 == 0 (SP_ERR_UNSUPPORTED otherwise).
 * Synchronises `stream` once (the total size sizes the buffer).  On success *out
 * is a new handle owning its device buffers; on error *out is NULL and nothing
 * is leaked.  Inputs are only read and may be freed once the call returns. */
sp_status sp_compress(const void* w_dev, const uint8_t* mask_dev, int64_t n, int64_t k, sp_dtype dtype,
                      const float* scale_dev, sp_alloc_fn alloc, sp_free_fn free_fn, void* alloc_ctx,
                      void* stream, sp_matrix** out);

/* Expand the handle back to the dense masked weight (the inverse of the Sec. 2.4.2 storage:
 * each submatrix's values placed by its bitmask, Sec. 2.4.1): w_out_dev [N, K] of the
 * handle's dtype (int8 values without their scales for SP_INT8), zero where masked
 * out, bit-exact.  Asynchronous on `stream`; w_out_dev is caller-owned.
 * SP_ERR_BAD_HANDLE for a dead handle, SP_ERR_INVALID_ARG for a null output. */
sp_status sp_decompress(const sp_matrix* h, void* w_out_dev, void* stream);

/* Bytes of device workspace that sp_linear needs for a batch of m rows (its split-K scratch;
 * library plumbing with no counterpart in the paper), written to *bytes (0 for m == 0).  Host only.  SP_ERR_INVALID_ARG for m < 0 or a null `bytes`. */
sp_status sp_workspace_size(const sp_matrix* h, int64_t m, size_t* bytes);

/* y = x . (W o Mask)^T, FP32 accumulation, bf16 output (round to nearest even): the sparse
 * product of Sec. 2.4.2, the compressed submatrices streamed from global memory and expanded
 * on chip by their bitmasks; equal to the dense product with the masked weight.
 *   x_dev      [m, K] bf16.      y_dev [m, N] bf16 (fully overwritten).
 *   workspace  device memory of at least sp_workspace_size(h, m) bytes, zero-filled
 *              before its first use; every call leaves it ready for the next one.
 *              Calls that share a workspace must be ordered on one stream.
 *   m == 0 returns SP_OK without a launch.  No allocation, no host sync: the call
 *   can be captured in a CUDA graph.  Results are bitwise repeatable for a given
 *   (matrix, m, device). */
sp_status sp_linear(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* workspace_dev,
                    size_t workspace_bytes, void* stream);

/* sp_linear (Sec. 2.4.2) with an explicit kernel family (tests run each family on its own). */
sp_status sp_linear_ex(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* workspace_dev,
                       size_t workspace_bytes, sp_path path, void* stream);

/* Kernels that sp_linear_ex can launch (reported by sp_launch_count). */
enum {
  SP_KERNEL_NONE = 0,
  SP_KERNEL_CC_THREAD_PER_ROW = 1,  /* linear_cc_kernel: four warps share a chunk, thread = row */
  SP_KERNEL_CC_WARP_PER_CHUNK = 2,  /* linear_ccw_kernel (M <= 4): a warp per chunk, lane = 4 rows */
  SP_KERNEL_TENSOR_CORE = 3         /* linear_tc_kernel */
};

/* (Library plumbing; no counterpart in the paper.)  Number of kernel launches that
 * sp_linear_ex(h, x, m, y, ws, ws_bytes, path, stream)
 * makes, written to *launches: 0 for m == 0, one per 16 batch rows on the CUDA-core
 * family, one on the tensor-core family; if `kernel` is not null, the SP_KERNEL_* value
 * of the kernel used for the first 16 rows (or all rows) goes there.  For callers that
 * count launches or label profiles.  Host only: no GPU work.  SP_ERR_BAD_HANDLE for a
 * dead handle, SP_ERR_INVALID_ARG for m < 0, an unknown path or a null `launches`. */
sp_status sp_launch_count(const sp_matrix* h, int64_t m, sp_path path, int64_t* launches, int32_t* kernel);

/* sp_linear for callers that may not allocate device memory (the paper has no
 * counterpart; this is a deployment convenience).  Some callers receive only their
 * input and output buffers from a host framework or plugin interface that owns all
 * device memory, and some run latency-critical loops where cudaMalloc/cudaFree would
 * synchronise the device: neither can supply sp_linear's workspace.  This call runs the
 * CUDA-core decode kernel in its stream-K configuration, using instead a scratch array
 * of 16 MiB that the library keeps on every GPU that loads it (held until the process
 * exits).  It calls no cudaMalloc, cudaFree or other allocating routine.
 *   x_dev [m, K] bf16, y_dev [m, N] bf16, as for sp_linear.
 *   Returns SP_ERR_WORKSPACE if the kernel would need more scratch than the array holds.
 *   The first call on a device looks up the array's device address (set-up, once per
 *   device, with that device current); make that first call before any stream capture.
 *   The address is kept for the life of the process, so a device reset (cudaDeviceReset)
 *   between calls is not supported.
 *   Every call on a device shares the one array, and a call clears its arrival counters
 *   first: calls that overlap on the GPU (other streams, other threads) race and give
 *   wrong results; order them on one stream. */
sp_status sp_linear_noalloc(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* stream);

/* The masked weight step of sparse training (Sec. 2.1, Algorithm 1) applied in place to
 * the compressed form: every kept weight becomes
 *     w[n,k] <- bf16_rne(fma(-lr, grad[n,k], w[n,k]))      (float32, one rounding)
 * and masked-out weights stay zero, since the mask never changes.  Only the packed values
 * are rewritten; masks, chunk offsets, padding and the handle's metadata stay as they are,
 * so the handle stays valid for every other call.
 *   grad_dev   [N, K] float32, dense and row-major; the values of its masked-out
 *              entries are never used (they may hold anything, NaN included).
 *   lr         the step size, finite (SP_ERR_INVALID_ARG otherwise); 0 leaves the values
 *              unchanged.
 * bf16 handles only (SP_ERR_UNSUPPORTED for SP_INT8).  Asynchronous on `stream`; work
 * that reads the handle (sp_linear, sp_decompress, ...) must be ordered after it by the
 * caller, on the same stream or through an event.  The next sp_linear launch on the
 * handle then starts only once the update has finished (it is launched without
 * programmatic dependent launch, whose early start would let its first weight copies
 * read the values from before the update).  No allocation, no host sync.  Results are
 * bitwise deterministic. */
sp_status sp_masked_update(sp_matrix* h, const float* grad_dev, float lr, void* stream);

/* INT8 weights and INT8 activations (Sec. 3.4, the sparse INT8 deployment):
 *     y[m,n] = bf16_rne(sx[m] * sw[n] * sum_k qx[m,k] * qw[n,k] * Mask[n,k])
 * for a handle compressed from SP_INT8 values qw with per-row scales sw.  On GB300 the dense
 * INT8 tensor rate is far below the bf16 rate, so the activations are widened once,
 * x[m,k] = bf16_rne(qx[m,k] * sx[m]) (float32 product), into the workspace, and the
 * INT8-weight sparse linear of sp_linear runs on that x: FP32 accumulation, sw applied in
 * its epilogue, one bf16 rounding of y.
 *   qx_dev     [m, K] int8, row-major.        sx_dev [m] fp32 per-token scales.
 *   y_dev      [m, N] bf16 (fully overwritten).
 *   workspace  at least sp_w8a8_workspace_size(h, m) bytes, zero-filled before its first
 *              use: sp_linear's workspace for (h, m) followed by the widened activations,
 *              so one buffer can serve sp_linear and sp_linear_w8a8 calls ordered on one
 *              stream.
 * SP_ERR_UNSUPPORTED for a bf16 handle; otherwise the errors of sp_linear.  m == 0 returns
 * SP_OK without a launch.  Two launches (widening, linear), no allocation, no host sync. */
sp_status sp_linear_w8a8(const sp_matrix* h, const int8_t* qx_dev, const float* sx_dev, int64_t m, void* y_dev,
                         void* workspace_dev, size_t workspace_bytes, void* stream);

/* Workspace bytes sp_linear_w8a8 (Sec. 3.4) needs for a batch of m rows (0 for m == 0);
 * library plumbing with no counterpart in the paper.  Host only.
 * SP_ERR_INVALID_ARG for m < 0 or a null `bytes`, SP_ERR_BAD_HANDLE for a dead handle. */
sp_status sp_w8a8_workspace_size(const sp_matrix* h, int64_t m, size_t* bytes);

/* Failure-path test (the paper has no counterpart; nothing calls it in normal use).  Runs
 * sp_linear's CUDA-core decode kernel for m = 1..4 rows -- the warp-per-chunk kernel, as
 * sp_linear would -- with one consumer warp of its first CTA first waiting on a
 * shared-memory barrier that nothing completes and no copy targets.  That bounded wait gives
 * up after wait_ms milliseconds and records SP_ERR_TIMEOUT in the device status word, as any
 * expired wait does; the warp then goes on normally, so the launch ends and y is the product
 * sp_linear would give.  Afterwards sp_check() returns SP_ERR_TIMEOUT once (and clears the
 * status), and the workspace is ready for the next call.  Arguments as for sp_linear;
 * wait_ms in 1..10000 (SP_ERR_INVALID_ARG otherwise); SP_ERR_UNSUPPORTED when m is outside
 * 1..4, for an SP_INT8 handle, or when sp_linear would not run the warp-per-chunk kernel
 * for this matrix.  The waiting warp is compiled into a variant of the kernel of its own;
 * sp_linear never runs that variant. */
sp_status sp_test_expired_wait(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* workspace_dev,
                               size_t workspace_bytes, uint32_t wait_ms, void* stream);

/* (Library plumbing; no counterpart in the paper.)  A copy of the handle with its own
 * device buffers (same bytes), allocated on the
 * current device, which must be the handle's (SP_ERR_INVALID_ARG otherwise).  The copies
 * run on `stream`, which is synchronised before the call returns. */
sp_status sp_clone(const sp_matrix* h, sp_alloc_fn alloc, sp_free_fn free_fn, void* alloc_ctx, void* stream,
                   sp_matrix** out);

/* (Library plumbing; no counterpart in the paper.)  Release the handle and its device
 * buffers.  The caller must ensure no queued
 * work still reads them (e.g. synchronise the stream first).  NULL is a no-op. */
sp_status sp_free(sp_matrix* h);

/* (Library plumbing; no counterpart in the paper.)  Shape and storage facts of a live
 * handle (the Sec. 2.4.2 storage's sizes), written to *info (the fields of sp_info_t).
 * Host only, no GPU work.  SP_ERR_BAD_HANDLE for a dead handle, SP_ERR_INVALID_ARG for a
 * null `info`. */
sp_status sp_info(const sp_matrix* h, sp_info_t* info);

/* (Library plumbing; no counterpart in the paper.)  Synchronously copy the compressed
 * bytes (info.bytes) and the RB*T+1 chunk
 * offsets (uint64) to host memory; either destination may be NULL. */
sp_status sp_copy_out(const sp_matrix* h, void* buf_host, size_t buf_cap, uint64_t* off_host, size_t off_count);

/* (Library plumbing; no counterpart in the paper.)  Synchronise `stream`; report and clear
 * the current device's status word.
 * Returns SP_ERR_TIMEOUT if a kernel's bounded wait expired since the last
 * check, SP_ERR_CUDA if the stream reported an error, else SP_OK. */
sp_status sp_check(void* stream);

/* Static English name of a status code (library plumbing; no counterpart in the paper). */
const char* sp_status_string(sp_status s);

#ifdef __cplusplus
}
#endif

#endif /* SP_H */
