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
// kernel is laid out for it: one CTA per 128 x 64 chunk, warp w taking chunk rows
// 32w .. 32w+31, lane l the column pair (2l, 2l+1) of a row, so every row segment of the
// gradient (256 bytes) is one coalesced request; a pair whose two columns are masked out
// is not read.  A row's first value is a popc prefix over the chunk's 128 masks (one CTA
// scan), a column's value index the popcount of its row's mask below it.
#include "sp_internal.cuh"

namespace sp {
namespace {

constexpr int kUnroll = 8;                 // rows of one warp whose loads are in flight together

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }

__device__ __forceinline__ uint16_t float_to_bf16_bits_rne(float f) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

__global__ void __launch_bounds__(kRows) masked_update_kernel(uint8_t* __restrict__ buf,
                                                              const uint64_t* __restrict__ off,
                                                              const float* __restrict__ grad, float neg_lr,
                                                              int64_t N, int64_t K, int T) {
  __shared__ uint64_t s_mask[kRows];
  __shared__ int s_start[kRows];
  __shared__ int s_warp[kRows / 32];
  const int64_t c = blockIdx.x;
  const int64_t rb = c / T, t = c % T;
  const int r = threadIdx.x, lane = r & 31, warp = r >> 5;
  uint8_t* chunk = buf + off[c];
  uint16_t* vals = reinterpret_cast<uint16_t*>(chunk + kMaskBytes);

  // Row starts: exclusive prefix sum of the 128 rows' popcounts.
  const uint64_t m = reinterpret_cast<const uint64_t*>(chunk)[r];
  const int cnt = __popcll(m);
  int incl = cnt;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += u;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  int base = 0;
#pragma unroll
  for (int w = 0; w < kRows / 32; ++w)
    if (w < warp) base += s_warp[w];
  s_mask[r] = m;
  s_start[r] = base + incl - cnt;
  __syncthreads();

  // Lane l owns columns 2l and 2l+1 of every row the warp visits.
  const int j = 2 * lane;
  const uint64_t below = (1ull << j) - 1ull;  // j <= 62
  const int64_t col = (int64_t)kTileK * t + j;
  const int row0 = warp * 32;
#pragma unroll 1
  for (int i0 = 0; i0 < 32; i0 += kUnroll) {
    float2 g[kUnroll];
    uint16_t v0[kUnroll], v1[kUnroll];
    int pos[kUnroll];
    uint32_t two[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int rr = row0 + i0 + u;
      const uint64_t mr = s_mask[rr];
      const int64_t n = rb * kRows + rr;
      two[u] = (uint32_t)(mr >> j) & 3u;
      // A well-formed chunk has no bits in rows >= N or columns >= K; skip any such bit
      // rather than read past the gradient.
      const bool inside = n < N && col + ((two[u] >> 1) & 1u) < K;
      if (!inside) two[u] = 0;
      pos[u] = s_start[rr] + __popcll(mr & below);
      g[u] = make_float2(0.f, 0.f);
      v0[u] = 0;
      v1[u] = 0;
      if (two[u]) {
        g[u] = __ldcs(reinterpret_cast<const float2*>(grad + n * K + col));
        if (two[u] & 1u) {
          v0[u] = vals[pos[u]];
          if (two[u] & 2u) v1[u] = vals[pos[u] + 1];
        } else {
          v1[u] = vals[pos[u]];
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      if (two[u] & 1u) vals[pos[u]] = float_to_bf16_bits_rne(__fmaf_rn(neg_lr, g[u].x, bf16_bits_to_float(v0[u])));
      if (two[u] & 2u)
        vals[pos[u] + (two[u] & 1u)] =
            float_to_bf16_bits_rne(__fmaf_rn(neg_lr, g[u].y, bf16_bits_to_float(v1[u])));
    }
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace sp

using namespace sp;

extern "C" sp_status sp_masked_update(sp_matrix* h, const float* grad_dev, float lr, void* stream) {
  if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
  if (!grad_dev) return SP_ERR_INVALID_ARG;
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
  masked_update_kernel<<<(unsigned)C, kRows, 0, (cudaStream_t)stream>>>(h->d_buf, h->d_off, grad_dev, -lr, h->N,
                                                                          h->K, h->T);
  if (cudaGetLastError() != cudaSuccess) return SP_ERR_CUDA;
  return SP_OK;
}
