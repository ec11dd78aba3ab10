// sp_format.cu -- building and expanding the bitmask-compressed weight.
//
// sp_compress turns a dense weight plus keep-mask into the chunked format of
// include/sp.h (the submatrix storage of Sec. 2.4.2: dense nonzeros plus a
// bitmask per submatrix, with the per-block bitmask encoding of Sec. 2.4.1):
//   1. count:   one CTA per chunk, one thread per row: build the row's 64-bit
//               mask for the K-tile and count the kept entries of the chunk;
//   2. scan:    one CTA: exclusive scan of padded chunk sizes -> byte offsets;
//   3. (host)   read the total size, allocate the buffer;
//   4. scatter: one CTA per chunk: write the masks, a 128-row prefix sum of the
//               popcounts gives each row's first value slot, rows copy their kept
//               values in ascending column order, and the padding is zeroed.
// sp_decompress is the inverse (one CTA per chunk, one thread per row).
// None of this is on the timed path.
#include <algorithm>

#include "sp_internal.cuh"

namespace sp {
namespace {

__device__ __forceinline__ int block_excl_scan_128(int v, int* total, int* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    int u = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += u;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  int base = 0, all = 0;
#pragma unroll
  for (int w = 0; w < kRows / 32; ++w) {
    int s = s_warp[w];
    if (w < warp) base += s;
    all += s;
  }
  __syncthreads();
  *total = all;
  return base + incl - v;
}

// Also writes the chunk's quarter index (kept entries before rows 32, 64 and 96, and in the
// whole chunk; 16 bits each) and raises *max_quarter to its largest quarter count.
__global__ void __launch_bounds__(kRows) count_kernel(const uint8_t* __restrict__ mask, int64_t N, int64_t K, int T,
                                                      uint64_t* __restrict__ masks_out, int* __restrict__ cnt,
                                                      uint64_t* __restrict__ qidx, int* __restrict__ max_quarter) {
  __shared__ int s_warp[kRows / 32];
  __shared__ int s_q[kRows / 32];
  const int64_t c = blockIdx.x;
  const int64_t rb = c / T, t = c % T;
  const int r = threadIdx.x;
  const int64_t n = rb * kRows + r;
  uint64_t m = 0;
  if (n < N) {
    const int valid = (int)imin64((int64_t)kTileK, K - (int64_t)kTileK * t);  // multiple of 8
    const uint8_t* row = mask + n * K + (int64_t)kTileK * t;
    for (int g = 0; g < valid / 8; ++g) {
      const uint64_t v = *reinterpret_cast<const uint64_t*>(row + 8 * g);
#pragma unroll
      for (int b = 0; b < 8; ++b)
        if ((v >> (8 * b)) & 0xffu) m |= 1ull << (8 * g + b);
    }
  }
  masks_out[c * kRows + r] = m;
  int total;
  const int excl = block_excl_scan_128(__popcll(m), &total, s_warp);
  if ((r & 31) == 0) s_q[r >> 5] = excl;
  __syncthreads();
  if (r == 0) {
    cnt[c] = total;
    qidx[c] = (uint64_t)s_q[1] | ((uint64_t)s_q[2] << 16) | ((uint64_t)s_q[3] << 32) | ((uint64_t)total << 48);
    const int q = max(max(s_q[1] - s_q[0], s_q[2] - s_q[1]), max(s_q[3] - s_q[2], total - s_q[3]));
    atomicMax(max_quarter, q);
  }
}

// meta[0] = total bytes, meta[1] = largest chunk, meta[2] = kept entries
__global__ void __launch_bounds__(1024) scan_kernel(const int* __restrict__ cnt, int64_t C, int esize,
                                                    uint64_t* __restrict__ off, uint64_t* __restrict__ meta) {
  __shared__ uint64_t s_warp[32];
  __shared__ uint64_t s_max[32], s_nnz[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint64_t carry = 0, mx = 0, nnz = 0;
  for (int64_t base = 0; base < C; base += 1024) {
    const int64_t i = base + threadIdx.x;
    uint64_t sz = 0;
    if (i < C) {
      const uint64_t kept = (uint64_t)cnt[i];
      sz = (kMaskBytes + kept * esize + 15) / 16 * 16;
      mx = max(mx, sz);
      nnz += kept;
    }
    uint64_t incl = sz;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      uint64_t u = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += u;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    uint64_t wbase = 0, all = 0;
    for (int w = 0; w < 32; ++w) {
      if (w < warp) wbase += s_warp[w];
      all += s_warp[w];
    }
    if (i < C) off[i] = carry + wbase + incl - sz;
    carry += all;
    __syncthreads();
  }
  for (int d = 16; d > 0; d >>= 1) {
    mx = max(mx, __shfl_down_sync(0xffffffffu, mx, d));
    nnz += __shfl_down_sync(0xffffffffu, nnz, d);
  }
  if (lane == 0) {
    s_max[warp] = mx;
    s_nnz[warp] = nnz;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    uint64_t a = 0, b = 0;
    for (int w = 0; w < 32; ++w) {
      a = max(a, s_max[w]);
      b += s_nnz[w];
    }
    off[C] = carry;
    meta[0] = carry;
    meta[1] = a;
    meta[2] = b;
  }
}

__global__ void __launch_bounds__(kRows) scatter_kernel(const uint8_t* __restrict__ w, int esize, int64_t N, int64_t K,
                                                        int T, const uint64_t* __restrict__ masks,
                                                        const uint64_t* __restrict__ off, uint8_t* __restrict__ buf) {
  __shared__ int s_warp[kRows / 32];
  const int64_t c = blockIdx.x;
  const int64_t rb = c / T, t = c % T;
  const int r = threadIdx.x;
  const int64_t n = rb * kRows + r;
  uint8_t* chunk = buf + off[c];
  const uint64_t m = masks[c * kRows + r];
  reinterpret_cast<uint64_t*>(chunk)[r] = m;
  int total;
  const int e0 = block_excl_scan_128(__popcll(m), &total, s_warp);
  uint8_t* vals = chunk + kMaskBytes;
  if (m) {
    const uint8_t* row = w + (n * K + (int64_t)kTileK * t) * esize;
    uint64_t mm = m;
    int i = 0;
    while (mm) {
      const int j = __ffsll((long long)mm) - 1;
      mm &= mm - 1;
      if (esize == 2) {
        const uint16_t v = *reinterpret_cast<const uint16_t*>(row + 2 * j);
        *reinterpret_cast<uint16_t*>(vals + 2 * (e0 + i)) = v;
      } else {
        vals[e0 + i] = row[j];
      }
      ++i;
    }
  }
  const uint64_t used = kMaskBytes + (uint64_t)total * esize;
  const uint64_t size = off[c + 1] - off[c];
  for (uint64_t b = used + r; b < size; b += kRows) chunk[b] = 0;
}

__global__ void __launch_bounds__(kRows) decompress_kernel(const uint8_t* __restrict__ buf,
                                                           const uint64_t* __restrict__ off, int esize, int64_t N,
                                                           int64_t K, int T, uint8_t* __restrict__ out) {
  __shared__ int s_warp[kRows / 32];
  const int64_t c = blockIdx.x;
  const int64_t rb = c / T, t = c % T;
  const int r = threadIdx.x;
  const int64_t n = rb * kRows + r;
  const uint8_t* chunk = buf + off[c];
  const uint64_t m = reinterpret_cast<const uint64_t*>(chunk)[r];
  int total;
  const int e0 = block_excl_scan_128(__popcll(m), &total, s_warp);
  if (n >= N) return;
  const uint8_t* vals = chunk + kMaskBytes;
  const int valid = (int)imin64((int64_t)kTileK, K - (int64_t)kTileK * t);
  uint8_t* row = out + (n * K + (int64_t)kTileK * t) * esize;
  int i = 0;
  for (int j = 0; j < valid; ++j) {
    const bool kept = (m >> j) & 1u;
    if (esize == 2) {
      uint16_t v = 0;
      if (kept) v = *reinterpret_cast<const uint16_t*>(vals + 2 * (e0 + i));
      reinterpret_cast<uint16_t*>(row)[j] = v;
    } else {
      row[j] = kept ? vals[e0 + i] : 0;
    }
    i += kept;
  }
}

}  // namespace

void* dev_alloc(const sp_matrix* h, size_t bytes) {
  if (bytes == 0) bytes = 16;
  if (h->alloc) return h->alloc(bytes, h->ctx);
  void* p = nullptr;
  if (cudaMalloc(&p, bytes) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}

void dev_free(const sp_matrix* h, void* p) {
  if (!p) return;
  if (h->free_fn)
    h->free_fn(p, h->ctx);
  else
    cudaFree(p);
}

sp_status launch_compress(const void* w, const uint8_t* mask, int64_t N, int64_t K, sp_dtype dt, const float* scale,
                          sp_alloc_fn alloc, sp_free_fn free_fn, void* ctx, cudaStream_t stream, sp_matrix** out) {
  sp_matrix* h = new sp_matrix();
  h->magic = 0;
  h->N = N;
  h->K = K;
  h->T = (int32_t)((K + kTileK - 1) / kTileK);
  h->RB = (int32_t)((N + kRows - 1) / kRows);
  h->dtype = dt;
  h->esize = dt == SP_BF16 ? 2 : 1;
  h->alloc = alloc;
  h->free_fn = free_fn;
  h->ctx = ctx;
  cudaGetDevice(&h->device);
  cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  const int64_t C = (int64_t)h->RB * h->T;

  sp_status st = SP_OK;
  uint64_t* d_masks = (uint64_t*)dev_alloc(h, (size_t)C * kRows * sizeof(uint64_t));
  int* d_cnt = (int*)dev_alloc(h, (size_t)C * sizeof(int));
  uint64_t* d_meta = (uint64_t*)dev_alloc(h, 4 * sizeof(uint64_t));
  h->d_off = (uint64_t*)dev_alloc(h, (size_t)(C + 1) * sizeof(uint64_t));
  h->d_qidx = (uint64_t*)dev_alloc(h, (size_t)C * sizeof(uint64_t));
  uint64_t meta[4] = {0, 0, 0, 0};
  if (!d_masks || !d_cnt || !d_meta || !h->d_off || !h->d_qidx) {
    st = SP_ERR_OUT_OF_MEMORY;
    goto fail;
  }
  // meta[3] holds the largest quarter count (count_kernel's atomicMax target)
  if (cudaMemsetAsync(d_meta, 0, 4 * sizeof(uint64_t), stream) != cudaSuccess) {
    st = SP_ERR_CUDA;
    goto fail;
  }
  count_kernel<<<(unsigned)C, kRows, 0, stream>>>(mask, N, K, h->T, d_masks, d_cnt, h->d_qidx,
                                                   reinterpret_cast<int*>(d_meta + 3));
  scan_kernel<<<1, 1024, 0, stream>>>(d_cnt, C, h->esize, h->d_off, d_meta);
  if (cudaGetLastError() != cudaSuccess) {
    st = SP_ERR_CUDA;
    goto fail;
  }
  if (cudaMemcpyAsync(meta, d_meta, sizeof(meta), cudaMemcpyDeviceToHost, stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    st = SP_ERR_CUDA;
    goto fail;
  }
  h->bytes = meta[0];
  h->max_chunk = meta[1];
  h->nnz = (int64_t)meta[2];
  h->max_quarter = (uint32_t)(meta[3] & 0xffffffffu);
  h->d_buf = (uint8_t*)dev_alloc(h, (size_t)std::max<uint64_t>(h->bytes, 16));
  if (!h->d_buf) {
    st = SP_ERR_OUT_OF_MEMORY;
    goto fail;
  }
  if (dt == SP_INT8) {
    h->d_scale = (float*)dev_alloc(h, (size_t)N * sizeof(float));
    if (!h->d_scale) {
      st = SP_ERR_OUT_OF_MEMORY;
      goto fail;
    }
    if (cudaMemcpyAsync(h->d_scale, scale, (size_t)N * sizeof(float), cudaMemcpyDeviceToDevice, stream) !=
        cudaSuccess) {
      st = SP_ERR_CUDA;
      goto fail;
    }
  }
  scatter_kernel<<<(unsigned)C, kRows, 0, stream>>>((const uint8_t*)w, h->esize, N, K, h->T, d_masks, h->d_off,
                                                     h->d_buf);
  if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(stream) != cudaSuccess) {
    st = SP_ERR_CUDA;
    goto fail;
  }
  dev_free(h, d_masks);
  dev_free(h, d_cnt);
  dev_free(h, d_meta);
  h->magic = SP_MAGIC;
  *out = h;
  return SP_OK;

fail:
  cudaStreamSynchronize(stream);
  cudaGetLastError();
  dev_free(h, d_masks);
  dev_free(h, d_cnt);
  dev_free(h, d_meta);
  dev_free(h, h->d_off);
  dev_free(h, h->d_qidx);
  dev_free(h, h->d_buf);
  dev_free(h, h->d_scale);
  delete h;
  return st;
}

sp_status launch_decompress(const sp_matrix* h, void* w_out, cudaStream_t stream) {
  const int64_t C = (int64_t)h->RB * h->T;
  decompress_kernel<<<(unsigned)C, kRows, 0, stream>>>(h->d_buf, h->d_off, h->esize, h->N, h->K, h->T,
                                                        (uint8_t*)w_out);
  return cudaGetLastError() == cudaSuccess ? SP_OK : SP_ERR_CUDA;
}

}  // namespace sp
