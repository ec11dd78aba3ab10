// sp_stack.cu -- elementwise glue of the linear-stack decode step (include/sp_stack.h).
// Each thread moves 8 bf16 (16 bytes) per access; FP32 arithmetic, one RNE rounding.
// Launched with programmatic dependent launch, like the sparse linears around them: a
// kernel's CTAs become resident while the previous grid runs and read nothing before
// griddepcontrol.wait (which returns once every earlier grid of the stream has completed).
// At M = 1 a glue kernel releases the next launch at once, so the next linear's CTAs
// become resident and copy weights while the glue runs; at M > 1 the release comes with
// the glue's exit.  Measured on GB300 (graph of the 32-layer step, 70%): early release
// 450 / 1277 tok/s at M = 1 / 4 (bf16), release at exit 432 / 1358, no PDL 446 / 1144;
// the M = 1 linears run six CTAs per SM and gain from early residency, the four-per-SM
// M > 1 linears lose by it (their CTAs land unevenly in the slots the previous linear's
// tail leaves).
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

__device__ __forceinline__ void glue_begin(bool early_release) {
  pdl_wait();
  if (early_release) pdl_launch_dependents();
}

__global__ void copy_columns_kernel(uint4* __restrict__ out, const uint4* __restrict__ in, int64_t M,
                                    int64_t in_stride8, int64_t col8, int64_t ncols8, bool early_release) {
  glue_begin(early_release);
  const int64_t total = M * ncols8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = i / ncols8, j = i % ncols8;
    out[i] = in[m * in_stride8 + col8 + j];
  }
}

__global__ void residual_add_kernel(uint4* __restrict__ h, const uint4* __restrict__ a, const uint4* __restrict__ r,
                                    int64_t M, int64_t n8, bool early_release) {
  glue_begin(early_release);
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

__global__ void mul_halves_kernel(uint4* __restrict__ out, const uint4* __restrict__ g, int64_t M, int64_t f8,
                                  bool early_release) {
  glue_begin(early_release);
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

// out[m, j] = bf16(g[m, 2j] * g[m, 2j + 1]): eight outputs per thread from two 16-byte
// loads of g (interleaved gate/up rows' outputs).
__global__ void mul_pairs_kernel(uint4* __restrict__ out, const uint4* __restrict__ g, int64_t M, int64_t f8,
                                 bool early_release) {
  glue_begin(early_release);
  const int64_t total = M * f8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = i / f8, j = i % f8;
    const uint4 a = g[m * 2 * f8 + 2 * j], b = g[m * 2 * f8 + 2 * j + 1];
    uint4 o;
    o.x = pack2(lo_f(a.x) * hi_f(a.x), lo_f(a.y) * hi_f(a.y));
    o.y = pack2(lo_f(a.z) * hi_f(a.z), lo_f(a.w) * hi_f(a.w));
    o.z = pack2(lo_f(b.x) * hi_f(b.x), lo_f(b.y) * hi_f(b.y));
    o.w = pack2(lo_f(b.z) * hi_f(b.z), lo_f(b.w) * hi_f(b.w));
    out[i] = o;
  }
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

template <typename... Params, typename... Args>
sp_status launch_glue(void (*kern)(Params...), int64_t total, cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  int64_t b = (total + kBlock - 1) / kBlock;
  cfg.gridDim = dim3((unsigned)(b < 1 ? 1 : b > 4096 ? 4096 : b));
  cfg.blockDim = dim3(kBlock);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, kern, args...) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  return SP_OK;
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
  return launch_glue(copy_columns_kernel, M * ncols / 8, (cudaStream_t)stream, (uint4*)out, (const uint4*)in, M,
                     in_stride / 8, col0 / 8, ncols / 8, M == 1);
}

sp_status sp_residual_add(void* h, const void* a, const void* r, int64_t M, int64_t N, void* stream) {
  if (!h || !a || !r || M < 0 || N < 0) return SP_ERR_INVALID_ARG;
  if (N % 8) return SP_ERR_UNSUPPORTED;
  if (!al16(h) || !al16(a) || !al16(r)) return SP_ERR_ALIGNMENT;
  if (M == 0 || N == 0) return SP_OK;
  return launch_glue(residual_add_kernel, M * N / 8, (cudaStream_t)stream, (uint4*)h, (const uint4*)a,
                     (const uint4*)r, M, N / 8, M == 1);
}

sp_status sp_mul_halves(void* out, const void* g, int64_t M, int64_t F, void* stream) {
  if (!out || !g || M < 0 || F < 0) return SP_ERR_INVALID_ARG;
  if (F % 8) return SP_ERR_UNSUPPORTED;
  if (!al16(out) || !al16(g)) return SP_ERR_ALIGNMENT;
  if (M == 0 || F == 0) return SP_OK;
  return launch_glue(mul_halves_kernel, M * F / 8, (cudaStream_t)stream, (uint4*)out, (const uint4*)g, M, F / 8,
                     M == 1);
}

sp_status sp_mul_pairs(void* out, const void* g, int64_t M, int64_t F, void* stream) {
  if (!out || !g || M < 0 || F < 0) return SP_ERR_INVALID_ARG;
  if (F % 8) return SP_ERR_UNSUPPORTED;
  if (!al16(out) || !al16(g)) return SP_ERR_ALIGNMENT;
  if (M == 0 || F == 0) return SP_OK;
  return launch_glue(mul_pairs_kernel, M * F / 8, (cudaStream_t)stream, (uint4*)out, (const uint4*)g, M, F / 8,
                     M == 1);
}

}  // extern "C"
