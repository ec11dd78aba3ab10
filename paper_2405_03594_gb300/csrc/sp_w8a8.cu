// sp_w8a8.cu -- sp_linear_w8a8: INT8 weights and INT8 activations (Sec. 3.4, the sparse
// INT8 deployment), y[m, n] = sx[m] * sw[n] * sum_k qx[m, k] * qw[n, k] * Mask[n, k].
//
// The paper's CPU engine runs this product in integer arithmetic (VNNI).  On GB300 the
// dense INT8 tensor rate is far below the bf16 rate, so INT8 is not a fast path there;
// what INT8 activations bring is their format.  The call therefore widens the activations
// once, x[m, k] = bf16_rne(qx[m, k] * sx[m]) (float32 product, one rounding), into the
// caller's workspace, and runs the INT8-weight sparse linear on that x (its epilogue
// applies sw[n]).  The widening is one elementwise pass over M x K bytes; every kernel
// choice of sp_linear (CUDA-core decode, tensor-core prefill) applies unchanged.  The
// widening runs under programmatic dependent launch like the linears: it writes x only after
// griddepcontrol.wait (every earlier grid of the stream has completed), and it releases the
// linear that follows at once for one-row batches (whose six-CTA launch then copies its
// weights while the widening runs) and at its exit otherwise, as the stack's glue kernels do.
#include <algorithm>

#include "sp_internal.cuh"

namespace sp {
namespace {

constexpr int kWidenBlock = 256;

// Eight activations per thread: one 8-byte load of qx, one 16-byte store of bf16.
// K % 8 == 0 (checked at compression), so a row holds K / 8 whole groups.
__global__ void __launch_bounds__(kWidenBlock) widen_kernel(const uint2* __restrict__ qx, const float* __restrict__ sx,
                                                            uint4* __restrict__ x, int64_t M, int64_t k8,
                                                            bool early_release) {
  pdl_wait();
  if (early_release) pdl_launch_dependents();
  const int64_t total = M * k8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const float s = sx[i / k8];
    const uint2 q = qx[i];
    uint32_t w[4];
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const uint32_t src = p < 2 ? q.x : q.y;
      const int sh = (p & 1) * 16;
      const float a = (float)(int8_t)((src >> sh) & 0xffu) * s;
      const float b = (float)(int8_t)((src >> (sh + 8)) & 0xffu) * s;
      w[p] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(a)) |
             ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(b)) << 16);
    }
    x[i] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t round256(size_t b) { return (b + 255) / 256 * 256; }

}  // namespace
}  // namespace sp

using namespace sp;

// Workspace layout: [sp_linear's workspace for (h, m)][widened x: m x K bf16].  sp_linear's
// part starts with its arrival counters at a fixed offset, so a buffer shared with plain
// sp_linear calls (and with w8a8 calls of other batch sizes) never has widened activations
// written over the counters.
extern "C" sp_status sp_w8a8_workspace_size(const sp_matrix* h, int64_t m, size_t* bytes) {
  if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
  if (!bytes || m < 0) return SP_ERR_INVALID_ARG;
  size_t lin = 0;
  const sp_status st = sp_workspace_size(h, m, &lin);
  if (st != SP_OK) return st;
  *bytes = m == 0 ? 0 : round256(lin) + round256((size_t)m * (size_t)h->K * 2);
  return SP_OK;
}

extern "C" sp_status sp_linear_w8a8(const sp_matrix* h, const int8_t* qx_dev, const float* sx_dev, int64_t m,
                                    void* y_dev, void* workspace_dev, size_t workspace_bytes, void* stream) {
  if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
  if (h->dtype != SP_INT8) return SP_ERR_UNSUPPORTED;
  if (m < 0) return SP_ERR_INVALID_ARG;
  if (m == 0) return SP_OK;
  if (!qx_dev || !sx_dev || !y_dev) return SP_ERR_INVALID_ARG;
  if (!aligned16(qx_dev) || !aligned16(sx_dev) || !aligned16(y_dev) || (workspace_dev && !aligned16(workspace_dev)))
    return SP_ERR_ALIGNMENT;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;
  size_t lin = 0, need = 0;
  sp_status st = sp_workspace_size(h, m, &lin);
  if (st == SP_OK) st = sp_w8a8_workspace_size(h, m, &need);
  if (st != SP_OK) return st;
  if (!workspace_dev || workspace_bytes < need) return SP_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(workspace_dev);
  uint4* x = reinterpret_cast<uint4*>(ws + round256(lin));
  const int64_t k8 = h->K / 8;  // K % 8 == 0 (checked at compression)
  const int64_t total = m * k8;
  const int64_t blocks = std::max<int64_t>(
      1, std::min<int64_t>((total + kWidenBlock - 1) / kWidenBlock, (int64_t)h->num_sms * 8));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(kWidenBlock);
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, widen_kernel, reinterpret_cast<const uint2*>(qx_dev), sx_dev, x, m, k8, m == 1) !=
      cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  return sp_linear(h, x, m, y_dev, ws, round256(lin), stream);
}
