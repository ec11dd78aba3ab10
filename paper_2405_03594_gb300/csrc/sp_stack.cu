// sp_stack.cu -- elementwise glue of the linear-stack decode step (include/sp_stack.h).
// Each thread moves 8 bf16 (16 bytes) per access; FP32 arithmetic, one RNE rounding.
#include "../../include/sp_stack.h"
#include "sp_internal.cuh"

namespace sp {
namespace {

constexpr int kBlock = 256;

__device__ __forceinline__ float lo_f(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_f(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  return (uint32_t)float_to_bf16_bits_rn(a) | ((uint32_t)float_to_bf16_bits_rn(b) << 16);
}

__global__ void copy_columns_kernel(uint4* __restrict__ out, const uint4* __restrict__ in, int64_t M,
                                    int64_t in_stride8, int64_t col8, int64_t ncols8) {
  const int64_t total = M * ncols8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = i / ncols8, j = i % ncols8;
    out[i] = in[m * in_stride8 + col8 + j];
  }
}

__global__ void residual_add_kernel(uint4* __restrict__ h, const uint4* __restrict__ a, const uint4* __restrict__ r,
                                    int64_t M, int64_t n8) {
  const int64_t total = M * n8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const uint4 hv = h[i], av = a[i], rv = r[i % n8];
    uint4 o;
    o.x = pack2(lo_f(hv.x) + lo_f(av.x) + lo_f(rv.x), hi_f(hv.x) + hi_f(av.x) + hi_f(rv.x));
    o.y = pack2(lo_f(hv.y) + lo_f(av.y) + lo_f(rv.y), hi_f(hv.y) + hi_f(av.y) + hi_f(rv.y));
    o.z = pack2(lo_f(hv.z) + lo_f(av.z) + lo_f(rv.z), hi_f(hv.z) + hi_f(av.z) + hi_f(rv.z));
    o.w = pack2(lo_f(hv.w) + lo_f(av.w) + lo_f(rv.w), hi_f(hv.w) + hi_f(av.w) + hi_f(rv.w));
    h[i] = o;
  }
}

__global__ void mul_halves_kernel(uint4* __restrict__ out, const uint4* __restrict__ g, int64_t M, int64_t f8) {
  const int64_t total = M * f8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = i / f8, j = i % f8;
    const uint4 a = g[m * 2 * f8 + j], b = g[m * 2 * f8 + f8 + j];
    uint4 o;
    o.x = pack2(lo_f(a.x) * lo_f(b.x), hi_f(a.x) * hi_f(b.x));
    o.y = pack2(lo_f(a.y) * lo_f(b.y), hi_f(a.y) * hi_f(b.y));
    o.z = pack2(lo_f(a.z) * lo_f(b.z), hi_f(a.z) * hi_f(b.z));
    o.w = pack2(lo_f(a.w) * lo_f(b.w), hi_f(a.w) * hi_f(b.w));
    out[i] = o;
  }
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

unsigned grid_for(int64_t total) {
  int64_t b = (total + kBlock - 1) / kBlock;
  if (b < 1) b = 1;
  if (b > 4096) b = 4096;
  return (unsigned)b;
}

}  // namespace
}  // namespace sp

using namespace sp;

extern "C" {

sp_status sp_copy_columns(void* out, const void* in, int64_t M, int64_t in_stride, int64_t col0, int64_t ncols,
                          void* stream) {
  if (!out || !in || M < 0 || ncols < 0 || col0 < 0 || in_stride < col0 + ncols) return SP_ERR_INVALID_ARG;
  if (ncols % 8 || col0 % 8 || in_stride % 8) return SP_ERR_UNSUPPORTED;
  if (!al16(out) || !al16(in)) return SP_ERR_ALIGNMENT;
  if (M == 0 || ncols == 0) return SP_OK;
  copy_columns_kernel<<<grid_for(M * ncols / 8), kBlock, 0, (cudaStream_t)stream>>>(
      (uint4*)out, (const uint4*)in, M, in_stride / 8, col0 / 8, ncols / 8);
  return cudaGetLastError() == cudaSuccess ? SP_OK : SP_ERR_CUDA;
}

sp_status sp_residual_add(void* h, const void* a, const void* r, int64_t M, int64_t N, void* stream) {
  if (!h || !a || !r || M < 0 || N < 0) return SP_ERR_INVALID_ARG;
  if (N % 8) return SP_ERR_UNSUPPORTED;
  if (!al16(h) || !al16(a) || !al16(r)) return SP_ERR_ALIGNMENT;
  if (M == 0 || N == 0) return SP_OK;
  residual_add_kernel<<<grid_for(M * N / 8), kBlock, 0, (cudaStream_t)stream>>>((uint4*)h, (const uint4*)a,
                                                                                (const uint4*)r, M, N / 8);
  return cudaGetLastError() == cudaSuccess ? SP_OK : SP_ERR_CUDA;
}

sp_status sp_mul_halves(void* out, const void* g, int64_t M, int64_t F, void* stream) {
  if (!out || !g || M < 0 || F < 0) return SP_ERR_INVALID_ARG;
  if (F % 8) return SP_ERR_UNSUPPORTED;
  if (!al16(out) || !al16(g)) return SP_ERR_ALIGNMENT;
  if (M == 0 || F == 0) return SP_OK;
  mul_halves_kernel<<<grid_for(M * F / 8), kBlock, 0, (cudaStream_t)stream>>>((uint4*)out, (const uint4*)g, M, F / 8);
  return cudaGetLastError() == cudaSuccess ? SP_OK : SP_ERR_CUDA;
}

}  // extern "C"
