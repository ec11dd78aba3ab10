// sp_noalloc.cu -- sp_linear_noalloc: the decode-batch sparse linear for callers that
// may not allocate device memory.
//
// Some callers are handed their input and output buffers by a host framework (a
// plugin or operator interface that owns every allocation) and are not allowed to
// allocate device memory of their own; others run in latency-critical loops where a
// cudaMalloc/cudaFree would synchronise the device.  They cannot provide the
// workspace that sp_linear needs.  This entry point runs the CUDA-core decode kernel in
// its stream-K configuration, with its scratch (the split-K arrival counters and FP32
// partials) in one fixed device array owned by the library, so it never calls
// cudaMalloc, cudaFree or any allocating routine.
//
// The array is a file-scope __device__ variable: every GPU that loads libsp holds its
// kNoAllocScratchBytes until the process exits.  In host code its name is only a
// host-side stand-in, so its device address is looked up with cudaGetSymbolAddress,
// once per device with that device current, on the first call made on that device.
#include <mutex>

#include "sp_internal.cuh"

namespace sp {
namespace {

constexpr size_t kNoAllocScratchBytes = 16u << 20;  // 16 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

void* g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

// Device address of this device's scratch array (set-up on first use per device).
sp_status scratch_address(int dev, void** out) {
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* ptr = nullptr;
    const cudaError_t rc = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (rc != cudaSuccess || ptr == nullptr) {
      cudaGetLastError();
      return SP_ERR_CUDA;
    }
    g_scratch_addr[dev] = ptr;
  }
  *out = g_scratch_addr[dev];
  return SP_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace sp

using namespace sp;

extern "C" sp_status sp_linear_noalloc(const sp_matrix* h, const void* x_dev, int64_t m, void* y_dev,
                                       void* stream) {
  if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
  if (m < 0) return SP_ERR_INVALID_ARG;
  if (m == 0) return SP_OK;
  if (!x_dev || !y_dev) return SP_ERR_INVALID_ARG;
  if (!aligned16(x_dev) || !aligned16(y_dev)) return SP_ERR_ALIGNMENT;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;
  if (dev < 0 || dev >= kMaxDevices) return SP_ERR_UNSUPPORTED;
  // The scratch must hold what sp_linear's workspace would: reject anything larger.
  const size_t need = workspace_bytes_cc(h, m);
  if (need > kNoAllocScratchBytes) return SP_ERR_WORKSPACE;
  void* scratch = nullptr;
  const sp_status st = scratch_address(dev, &scratch);
  if (st != SP_OK) return st;
  // The array keeps whatever the previous call left: the arrival counters must start
  // at zero, so clear them (stream-ordered; no allocation).
  if (cudaMemsetAsync(scratch, 0, ws_counter_bytes(h->num_sms), (cudaStream_t)stream) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  // stream-K split-K with the partials and arrival counters in the static array
  return launch_linear_cc(h, static_cast<const uint16_t*>(x_dev), m, static_cast<uint16_t*>(y_dev), scratch,
                          kNoAllocScratchBytes, (cudaStream_t)stream, /*allow_cluster=*/false);
}
