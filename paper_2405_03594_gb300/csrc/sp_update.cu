// sp_update.cu -- sp_masked_update: the masked weight step of Algorithm 1 (Sec. 2.1)
// applied directly to the compressed form.
//
// Sparse pretraining and fine-tuning keep the pruning mask fixed: a step computes
// theta <- theta - lr * (grad o Mask), so masked-out weights stay zero and only the kept
// weights change.  In the bitmask format the kept weights are exactly the stored values,
// so the step rewrites the packed values in place and leaves masks, offsets, padding and
// the quarter index untouched; the matrix never has to be decompressed.
//
// Arithmetic per kept (n, k): w <- bf16_rne(fma(-lr, grad[n, k], w)) in float32, one
// fused multiply-add and one rounding.  The dense float32 gradient is the large stream
// (4 bytes per weight against ~0.7 bytes of compressed weight at 70 % sparsity), so the
// kernel is laid out for it: one CTA of 16 warps per 128 x 64 chunk, warp w taking chunk
// rows 8w .. 8w+7 and lane l the column pair (2l, 2l+1) of each, so every row segment of
// the gradient (256 bytes) is one coalesced request, and all eight are issued before the
// chunk's masks are read.  A row's first value is a popc prefix over the chunk's 128
// masks (one scan by the first four warps), a column's value index the popcount of its
// row's mask below it.
#include "sp_internal.cuh"

namespace sp {
namespace {

constexpr int kUpdThreads = 512;                       // 16 warps per chunk
constexpr int kUpdRowsPerWarp = kRows / (kUpdThreads / 32);  // 8 chunk rows per warp

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }

__device__ __forceinline__ uint16_t float_to_bf16_bits_rne(float f) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

// The gradient loads of a warp's 8 rows are issued first, before the masks arrive, so
// the gradient stream and the mask read overlap: a lane reads its column pair of every
// row inside the matrix whether or not the pair is kept (the whole float32 gradient is
// read; at 70 % sparsity ~6 % of its 32-byte sectors hold no kept column).
__global__ void __launch_bounds__(kUpdThreads, 2) masked_update_kernel(uint8_t* __restrict__ buf,
                                                                       const uint64_t* __restrict__ off,
                                                                       const float* __restrict__ grad, float neg_lr,
                                                                       int64_t N, int64_t K, int T) {
  __shared__ uint64_t s_mask[kRows];
  __shared__ int s_start[kRows];
  __shared__ int s_warp[kRows / 32];
  const int64_t c = blockIdx.x;
  const int64_t rb = c / T, t = c % T;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int j = 2 * lane;  // this lane's column pair (j, j + 1) of the tile
  const int64_t col = (int64_t)kTileK * t + j;
  const int row0 = warp * kUpdRowsPerWarp;

  float2 g[kUpdRowsPerWarp];
#pragma unroll
  for (int u = 0; u < kUpdRowsPerWarp; ++u) {
    const int64_t n = rb * kRows + row0 + u;
    g[u] = make_float2(0.f, 0.f);
    if (n < N && col + 1 < K) g[u] = __ldcs(reinterpret_cast<const float2*>(grad + n * K + col));
  }

  uint8_t* chunk = buf + off[c];
  uint16_t* vals = reinterpret_cast<uint16_t*>(chunk + kMaskBytes);
  // Row starts: exclusive prefix sum of the 128 rows' popcounts (warps 0-3, thread = row).
  if (tid < kRows) {
    const uint64_t m = reinterpret_cast<const uint64_t*>(chunk)[tid];
    const int cnt = __popcll(m);
    int incl = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += v;
    }
    if (lane == 31) s_warp[warp] = incl;
    s_mask[tid] = m;
    s_start[tid] = incl - cnt;  // within the warp; the warps before it are added below
  }
  __syncthreads();
  const uint64_t below = (1ull << j) - 1ull;  // j <= 62
  int base = 0;
#pragma unroll
  for (int w = 0; w < kRows / 32; ++w)
    if (w < row0 / 32) base += s_warp[w];

  // Per row: which of the lane's two columns are kept (bits 0-1: j, j + 1) and, above
  // them, the index of the first kept one among the chunk's values (< 128 * 64).
  uint32_t pp[kUpdRowsPerWarp];
  uint32_t v[kUpdRowsPerWarp];  // the pair's stored values: low half column j, high half j + 1
#pragma unroll
  for (int u = 0; u < kUpdRowsPerWarp; ++u) {
    const int rr = row0 + u;
    const uint64_t mr = s_mask[rr];
    const int64_t n = rb * kRows + rr;
    uint32_t two = (uint32_t)(mr >> j) & 3u;
    // A well-formed chunk has no bits in rows >= N or columns >= K; skip any such bit
    // rather than use a gradient entry that was not read.
    if (!(n < N && col + 1 < K)) two = 0;
    const uint32_t pos = (uint32_t)(base + s_start[rr] + __popcll(mr & below));
    pp[u] = pos << 2 | two;
    uint32_t lo = 0, hi = 0;
    if (two & 1u) lo = vals[pos];
    if (two & 2u) hi = vals[pos + (two & 1u)];
    v[u] = lo | (hi << 16);
  }
#pragma unroll
  for (int u = 0; u < kUpdRowsPerWarp; ++u) {
    const uint32_t two = pp[u] & 3u, pos = pp[u] >> 2;
    if (two & 1u) vals[pos] = float_to_bf16_bits_rne(__fmaf_rn(neg_lr, g[u].x, bf16_bits_to_float((uint16_t)v[u])));
    if (two & 2u)
      vals[pos + (two & 1u)] =
          float_to_bf16_bits_rne(__fmaf_rn(neg_lr, g[u].y, bf16_bits_to_float((uint16_t)(v[u] >> 16))));
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace sp

using namespace sp;

extern "C" sp_status sp_masked_update(sp_matrix* h, const float* grad_dev, float lr, void* stream) {
  if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
  if (!grad_dev || !isfinite(lr)) return SP_ERR_INVALID_ARG;
  if (h->dtype != SP_BF16) return SP_ERR_UNSUPPORTED;
  if (!aligned16(grad_dev)) return SP_ERR_ALIGNMENT;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (dev != h->device) return SP_ERR_INVALID_ARG;
  const int64_t C = (int64_t)h->RB * h->T;  // < 2^31, checked by sp_compress
  if (h->nnz == 0) return SP_OK;
  masked_update_kernel<<<(unsigned)C, kUpdThreads, 0, (cudaStream_t)stream>>>(h->d_buf, h->d_off, grad_dev, -lr, h->N,
                                                                          h->K, h->T);
  if (cudaGetLastError() != cudaSuccess) return SP_ERR_CUDA;
  h->weights_written = 1;
  return SP_OK;
}
