// sp_api.cu -- the extern "C" surface of libsp (include/sp.h): argument checks,
// handle bookkeeping, kernel-family selection and the device status word.
#include <stdlib.h>

#include <algorithm>
#include <mutex>

#include "../../include/sp_stack.h"
#include "sp_internal.cuh"

namespace sp {

// One status word per device: kernels record the first expired bounded wait here.
__device__ int g_status_word;

namespace {
constexpr int kMaxDevices = 64;
int* g_status_ptr[kMaxDevices] = {};
std::mutex g_mu;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool live(const sp_matrix* h) { return h && h->magic == SP_MAGIC; }

// Largest batch that the CUDA-core family takes under SP_PATH_AUTO; larger batches go
// to the tensor-core family.  Measured crossover on the Llama-2-7B shapes at 70%: the
// CUDA-core path costs ~M FMAs per kept weight and the tensor-core path a fixed
// expansion per chunk, so the tensor cores win from M ~ 11 (bf16 values) and from
// M ~ 14 (int8 values, whose CUDA-core loop is cheaper and whose expansion costs more).
constexpr int64_t kCudaCoreMaxM_bf16 = 10;
constexpr int64_t kCudaCoreMaxM_int8 = 13;

bool uses_tensor_cores(const sp_matrix* h, int64_t m, sp_path path) {
  const int64_t cc_max = h->esize == 1 ? kCudaCoreMaxM_int8 : kCudaCoreMaxM_bf16;
  return path == SP_PATH_TENSOR_CORE || (path == SP_PATH_AUTO && m > cc_max);
}
}  // namespace

int* device_status_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    g_status_ptr[dev] = static_cast<int*>(p);
  }
  return g_status_ptr[dev];
}

uint64_t wait_timeout_ns() {
  static uint64_t ns = [] {
    const char* e = getenv("SP_WAIT_TIMEOUT_MS");
    long ms = e ? strtol(e, nullptr, 10) : 2000;
    if (ms <= 0) ms = 2000;
    return (uint64_t)ms * 1000000ull;
  }();
  return ns;
}

}  // namespace sp

using namespace sp;

extern "C" {

const char* sp_status_string(sp_status s) {
  switch (s) {
    case SP_OK: return "ok";
    case SP_ERR_INVALID_ARG: return "invalid argument";
    case SP_ERR_UNSUPPORTED: return "unsupported";
    case SP_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
    case SP_ERR_CUDA: return "CUDA error";
    case SP_ERR_OUT_OF_MEMORY: return "out of device memory";
    case SP_ERR_TIMEOUT: return "bounded device wait expired";
    case SP_ERR_BAD_HANDLE: return "bad handle";
    case SP_ERR_WORKSPACE: return "workspace missing or too small";
  }
  return "unknown status";
}

sp_status sp_compress(const void* w_dev, const uint8_t* mask_dev, int64_t n, int64_t k, sp_dtype dtype,
                      const float* scale_dev, sp_alloc_fn alloc, sp_free_fn free_fn, void* alloc_ctx, void* stream,
                      sp_matrix** out) {
  if (!out) return SP_ERR_INVALID_ARG;
  *out = nullptr;
  if (!w_dev || !mask_dev || n <= 0 || k <= 0) return SP_ERR_INVALID_ARG;
  if (dtype != SP_BF16 && dtype != SP_INT8) return SP_ERR_INVALID_ARG;
  if ((dtype == SP_INT8) != (scale_dev != nullptr)) return SP_ERR_INVALID_ARG;
  if ((alloc == nullptr) != (free_fn == nullptr)) return SP_ERR_INVALID_ARG;
  if (k % 8 != 0) return SP_ERR_UNSUPPORTED;
  if ((n + SP_CHUNK_ROWS - 1) / SP_CHUNK_ROWS * ((k + SP_TILE_K - 1) / SP_TILE_K) >= (int64_t)1 << 31)
    return SP_ERR_UNSUPPORTED;
  if (!aligned16(w_dev) || !aligned16(mask_dev) || (scale_dev && !aligned16(scale_dev))) return SP_ERR_ALIGNMENT;
  return launch_compress(w_dev, mask_dev, n, k, dtype, scale_dev, alloc, free_fn, alloc_ctx, (cudaStream_t)stream,
                         out);
}

sp_status sp_decompress(const sp_matrix* h, void* w_out_dev, void* stream) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (!w_out_dev) return SP_ERR_INVALID_ARG;
  if (!aligned16(w_out_dev)) return SP_ERR_ALIGNMENT;
  return launch_decompress(h, w_out_dev, (cudaStream_t)stream);
}

sp_status sp_workspace_size(const sp_matrix* h, int64_t m, size_t* bytes) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (!bytes || m < 0) return SP_ERR_INVALID_ARG;
  *bytes = m == 0 ? 0 : std::max(workspace_bytes_cc(h, m), workspace_bytes_tc(h, m));
  return SP_OK;
}

sp_status sp_linear_ex(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* workspace_dev,
                       size_t workspace_bytes, sp_path path, void* stream) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (m < 0) return SP_ERR_INVALID_ARG;
  if (path != SP_PATH_AUTO && path != SP_PATH_CUDA_CORE && path != SP_PATH_TENSOR_CORE) return SP_ERR_INVALID_ARG;
  if (m == 0) return SP_OK;
  if (!x_dev || !y_dev) return SP_ERR_INVALID_ARG;
  if (!aligned16(x_dev) || !aligned16(y_dev) || (workspace_dev && !aligned16(workspace_dev))) return SP_ERR_ALIGNMENT;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;
  // The documented contract, whatever kernel runs: a workspace of sp_workspace_size bytes.
  if (!workspace_dev || workspace_bytes < std::max(workspace_bytes_cc(h, m), workspace_bytes_tc(h, m)))
    return SP_ERR_WORKSPACE;
  if (uses_tensor_cores(h, m, path))
    return launch_linear_tc(h, static_cast<const uint16_t*>(x_dev), m, static_cast<uint16_t*>(y_dev), workspace_dev,
                            workspace_bytes, (cudaStream_t)stream);
  return launch_linear_cc(h, static_cast<const uint16_t*>(x_dev), m, static_cast<uint16_t*>(y_dev), workspace_dev,
                          workspace_bytes, (cudaStream_t)stream);
}

sp_status sp_linear_epi(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, int32_t epilogue,
                        const void* r_dev, void* workspace_dev, size_t workspace_bytes, void* stream) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (m < 0) return SP_ERR_INVALID_ARG;
  if (epilogue != SP_EPI_STORE && epilogue != SP_EPI_RESIDUAL && epilogue != SP_EPI_PAIR_PRODUCT)
    return SP_ERR_INVALID_ARG;
  if (epilogue == SP_EPI_RESIDUAL && !r_dev) return SP_ERR_INVALID_ARG;
  if (epilogue == SP_EPI_PAIR_PRODUCT && h->N % 2 != 0) return SP_ERR_INVALID_ARG;
  if (m == 0) return SP_OK;
  if (!x_dev || !y_dev) return SP_ERR_INVALID_ARG;
  if (!aligned16(x_dev) || !aligned16(y_dev) || (workspace_dev && !aligned16(workspace_dev)) ||
      (r_dev && (reinterpret_cast<uintptr_t>(r_dev) & 1u)))
    return SP_ERR_ALIGNMENT;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;
  if (!workspace_dev || workspace_bytes < std::max(workspace_bytes_cc(h, m), workspace_bytes_tc(h, m)))
    return SP_ERR_WORKSPACE;
  if (uses_tensor_cores(h, m, SP_PATH_AUTO)) return SP_ERR_UNSUPPORTED;
  return launch_linear_cc(h, static_cast<const uint16_t*>(x_dev), m, static_cast<uint16_t*>(y_dev), workspace_dev,
                          workspace_bytes, (cudaStream_t)stream, true, 0, epilogue,
                          static_cast<const uint16_t*>(r_dev));
}

sp_status sp_launch_count(const sp_matrix* h, int64_t m, sp_path path, int64_t* launches, int32_t* kernel) {
  if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
  if (m < 0 || !launches || (path != SP_PATH_AUTO && path != SP_PATH_CUDA_CORE && path != SP_PATH_TENSOR_CORE))
    return SP_ERR_INVALID_ARG;
  const bool tc = uses_tensor_cores(h, m, path);
  *launches = m == 0 ? 0 : tc ? 1 : (m + kMaxTokens - 1) / kMaxTokens;
  if (kernel) {
    if (m == 0)
      *kernel = SP_KERNEL_NONE;
    else if (tc)
      *kernel = SP_KERNEL_TENSOR_CORE;
    else
      *kernel = cc_kernel_kind(h, m) == 1 ? SP_KERNEL_CC_WARP_PER_CHUNK : SP_KERNEL_CC_THREAD_PER_ROW;
  }
  return SP_OK;
}

sp_status sp_linear(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* workspace_dev,
                    size_t workspace_bytes, void* stream) {
  return sp_linear_ex(h, x_dev, m, y_dev, workspace_dev, workspace_bytes, SP_PATH_AUTO, stream);
}

sp_status sp_test_expired_wait(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev, void* workspace_dev,
                               size_t workspace_bytes, uint32_t wait_ms, void* stream) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (!x_dev || !y_dev || wait_ms < 1 || wait_ms > 10000) return SP_ERR_INVALID_ARG;
  if (m < 1 || m > 4 || h->esize != 2 || cc_kernel_kind(h, m) != 1) return SP_ERR_UNSUPPORTED;
  if (!aligned16(x_dev) || !aligned16(y_dev) || (workspace_dev && !aligned16(workspace_dev))) return SP_ERR_ALIGNMENT;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;
  if (!workspace_dev || workspace_bytes < std::max(workspace_bytes_cc(h, m), workspace_bytes_tc(h, m)))
    return SP_ERR_WORKSPACE;
  return launch_linear_cc(h, static_cast<const uint16_t*>(x_dev), m, static_cast<uint16_t*>(y_dev), workspace_dev,
                          workspace_bytes, (cudaStream_t)stream, true, (uint64_t)wait_ms * 1000000ull);
}

sp_status sp_clone(const sp_matrix* h, sp_alloc_fn alloc, sp_free_fn free_fn, void* alloc_ctx, void* stream,
                   sp_matrix** out) {
  if (!out) return SP_ERR_INVALID_ARG;
  *out = nullptr;
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if ((alloc == nullptr) != (free_fn == nullptr)) return SP_ERR_INVALID_ARG;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;  // the copy lives on the source's device
  sp_matrix* c = new sp_matrix(*h);
  c->magic = 0;
  c->alloc = alloc;
  c->free_fn = free_fn;
  c->ctx = alloc_ctx;
  c->d_buf = nullptr;
  c->d_off = nullptr;
  c->d_qidx = nullptr;
  c->d_scale = nullptr;
  c->weights_written = 0;  // the copy below is synchronised
  const size_t off_bytes = ((size_t)h->RB * h->T + 1) * sizeof(uint64_t);
  cudaStream_t s = (cudaStream_t)stream;
  sp_status st = SP_OK;
  c->d_buf = (uint8_t*)dev_alloc(c, (size_t)std::max<uint64_t>(h->bytes, 16));
  c->d_off = (uint64_t*)dev_alloc(c, off_bytes);
  c->d_qidx = (uint64_t*)dev_alloc(c, off_bytes - sizeof(uint64_t));
  if (h->d_scale) c->d_scale = (float*)dev_alloc(c, (size_t)h->N * sizeof(float));
  if (!c->d_buf || !c->d_off || !c->d_qidx || (h->d_scale && !c->d_scale)) {
    st = SP_ERR_OUT_OF_MEMORY;
  } else if (cudaMemcpyAsync(c->d_buf, h->d_buf, h->bytes, cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
             cudaMemcpyAsync(c->d_off, h->d_off, off_bytes, cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
             cudaMemcpyAsync(c->d_qidx, h->d_qidx, off_bytes - sizeof(uint64_t), cudaMemcpyDeviceToDevice, s) !=
                 cudaSuccess ||
             (h->d_scale && cudaMemcpyAsync(c->d_scale, h->d_scale, (size_t)h->N * sizeof(float),
                                            cudaMemcpyDeviceToDevice, s) != cudaSuccess) ||
             cudaStreamSynchronize(s) != cudaSuccess) {
    st = SP_ERR_CUDA;
  }
  if (st != SP_OK) {
    cudaGetLastError();
    cudaStreamSynchronize(s);  // no copy may still target the buffers handed back below
    cudaGetLastError();
    dev_free(c, c->d_buf);
    dev_free(c, c->d_off);
    dev_free(c, c->d_qidx);
    dev_free(c, c->d_scale);
    delete c;
    return st;
  }
  c->magic = SP_MAGIC;
  *out = c;
  return SP_OK;
}

sp_status sp_free(sp_matrix* h) {
  if (!h) return SP_OK;
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  h->magic = 0;
  dev_free(h, h->d_buf);
  dev_free(h, h->d_off);
  dev_free(h, h->d_qidx);
  dev_free(h, h->d_scale);
  delete h;
  return SP_OK;
}

sp_status sp_info(const sp_matrix* h, sp_info_t* info) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (!info) return SP_ERR_INVALID_ARG;
  info->n = h->N;
  info->k = h->K;
  info->tiles = h->T;
  info->row_blocks = h->RB;
  info->dtype = h->dtype;
  info->device = h->device;
  info->nnz = h->nnz;
  info->bytes = h->bytes;
  info->max_chunk_bytes = h->max_chunk;
  info->scale_bytes = h->d_scale ? (uint64_t)h->N * 4 : 0;
  return SP_OK;
}

sp_status sp_copy_out(const sp_matrix* h, void* buf_host, size_t buf_cap, uint64_t* off_host, size_t off_count) {
  if (!live(h)) return SP_ERR_BAD_HANDLE;
  if (buf_host && buf_cap < h->bytes) return SP_ERR_INVALID_ARG;
  const size_t n_off = (size_t)h->RB * h->T + 1;
  if (off_host && off_count < n_off) return SP_ERR_INVALID_ARG;
  if (buf_host && cudaMemcpy(buf_host, h->d_buf, h->bytes, cudaMemcpyDeviceToHost) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (off_host && cudaMemcpy(off_host, h->d_off, n_off * sizeof(uint64_t), cudaMemcpyDeviceToHost) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  return SP_OK;
}

sp_status sp_check(void* stream) {
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  int* p = device_status_ptr();
  if (!p) return SP_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (v != 0) {
    const int zero = 0;
    cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice);
    return SP_ERR_TIMEOUT;
  }
  return SP_OK;
}

}  // extern "C"
