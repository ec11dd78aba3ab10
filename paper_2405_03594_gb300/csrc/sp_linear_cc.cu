// sp_linear_cc.cu -- decode-batch sparse linear on the CUDA cores.
//
// y[m, n] = sum_k x[m, k] * W[n, k] over the kept entries, read straight from the
// compressed chunks (Sec. 2.4.2: the compressed submatrices move from global
// memory onto the chip and are expanded there by their bitmask; decode is bound
// by those bytes, Sec. 2.4, 3.4).
//
// Launch: G persistent CTAs (2 per SM), each owning a contiguous run of chunks in
// storage order (stream-K), so every CTA streams one linear byte range.
//   warp 4, lane 0   producer: one cp.async.bulk per chunk (+ one 128-byte copy
//                    of x[m, 64t : 64t+64) per batch row) into a ring of
//                    `slots` shared-memory slots, each guarded by a full/empty
//                    mbarrier pair; weight bytes carry an L2 evict-first hint.
//   warps 0-3        consumers, thread r <-> row r of the chunk: its value slot
//                    is a popc prefix sum over the chunk's masks (warp scan plus
//                    the other warps' redux sums); it walks its set bits, gathers
//                    x[m, 64t+j] from registers of lane j%32 by shuffle, and
//                    accumulates in FP32.  At a row-block end the 128 rows are
//                    written (bf16, RNE), or -- when the row block is shared with
//                    other CTAs -- stored as an FP32 partial and summed in CTA
//                    order by the last CTA to arrive (deterministic split-K).
#include <algorithm>

#include "sp_internal.cuh"

namespace sp {
namespace {

constexpr int kConsumerWarps = 4;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kMaxTokens = 8;  // batch rows per launch of this kernel
constexpr int kMaxDevices = 64;
constexpr size_t kSmemBudget = 110 * 1024;  // ring slots; two CTAs share one SM
constexpr size_t kSmemOptIn = 112 * 1024;

template <int M, int ES>
__global__ void __launch_bounds__(kThreads, 2) linear_cc_kernel(const LinearParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)p.slots * p.slot_bytes);
  uint64_t* empty = full + p.slots;
  volatile int* s_flag = reinterpret_cast<volatile int*>(empty + p.slots);
  const int64_t w0 = range_begin(blockIdx.x, p.W, p.G);
  const int64_t w1 = range_begin(blockIdx.x + 1, p.W, p.G);
  const int T = p.T;

  if (tid == 0) {
    for (int s = 0; s < p.slots; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
    }
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int64_t it = 0;
      for (int64_t w = w0; w < w1; ++w, ++it) {
        const int s = (int)(it % p.slots);
        const uint32_t ph = (uint32_t)((it / p.slots) & 1);
        if (it >= p.slots && !mbar_wait(&empty[s], ph ^ 1u, p.timeout_ns)) {
          set_status(p.status, kStatusTimeout);
          break;
        }
        const int t = (int)(w % T);
        const uint64_t o0 = p.off[w];
        const uint32_t bytes = (uint32_t)(p.off[w + 1] - o0);
        const int valid = (int)imin64((int64_t)kTileK, p.K - (int64_t)kTileK * t);
        const uint32_t xb = (uint32_t)valid * 2u;
        uint8_t* slot = smem + (size_t)s * p.slot_bytes;
        mbar_arrive_expect_tx(&full[s], bytes + (uint32_t)M * xb);
        bulk_g2s_hint(slot, p.buf + o0, bytes, &full[s], pol);
#pragma unroll
        for (int m = 0; m < M; ++m)
          bulk_g2s(slot + p.chunk_region + m * 128, p.x + (int64_t)m * p.K + (int64_t)kTileK * t, xb, &full[s]);
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  float acc[M];
#pragma unroll
  for (int m = 0; m < M; ++m) acc[m] = 0.f;
  bool dead = false;  // a bounded wait expired: keep the barrier schedule, skip the math
  const int64_t rb_first = w0 / T;
  int64_t it = 0;
  for (int64_t w = w0; w < w1; ++w, ++it) {
    const int s = (int)(it % p.slots);
    const uint32_t ph = (uint32_t)((it / p.slots) & 1);
    if (!dead) {
      // the decision must be warp-uniform: the shuffles below use the full mask
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[s], ph, p.timeout_ns));
      if (!ok) {
        dead = true;
        set_status(p.status, kStatusTimeout);
      }
    }
    if (!dead) {
      const uint8_t* slot = smem + (size_t)s * p.slot_bytes;
      const uint64_t* masks = reinterpret_cast<const uint64_t*>(slot);
      uint64_t mk = masks[tid];
      const int pc = __popcll(mk);
      int incl = pc;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += u;
      }
      int base = 0;
      for (int k = 0; k < warp; ++k) base += (int)__reduce_add_sync(0xffffffffu, __popcll(masks[lane + 32 * k]));
      const int e0 = base + incl - pc;

      const uint16_t* xs = reinterpret_cast<const uint16_t*>(slot + p.chunk_region);
      uint32_t xr[M];
#pragma unroll
      for (int m = 0; m < M; ++m) xr[m] = (uint32_t)xs[m * 64 + lane] | ((uint32_t)xs[m * 64 + 32 + lane] << 16);

      const uint8_t* vals = slot + kMaskBytes + (size_t)e0 * ES;
      const int iters = (int)__reduce_max_sync(0xffffffffu, (unsigned)pc);
      for (int q = 0; q < iters; ++q) {
        const bool act = mk != 0;
        const int j = act ? (__ffsll((long long)mk) - 1) : 0;
        mk &= mk - 1;
        float wv = 0.f;
        if (act) {
          if (ES == 2)
            wv = bf16_bits_to_float(reinterpret_cast<const uint16_t*>(vals)[q]);
          else
            wv = (float)reinterpret_cast<const int8_t*>(vals)[q];
        }
        const int src = j & 31;
        const bool hi = j >= 32;
#pragma unroll
        for (int m = 0; m < M; ++m) {
          const uint32_t v = __shfl_sync(0xffffffffu, xr[m], src);
          const float xv = __uint_as_float(hi ? (v & 0xffff0000u) : (v << 16));
          if (act) acc[m] = fmaf(wv, xv, acc[m]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);

    // ------------------------------------------------------------ row-block end
    const int64_t rb = w / T;
    const int t = (int)(w % T);
    if (t != T - 1 && w + 1 != w1) continue;
    const int64_t seg_begin = rb * T;
    const int64_t n = rb * kRows + tid;
    const float sc = (ES == 1 && n < p.N) ? p.scale[n] : 1.f;
    if (seg_begin >= w0 && t == T - 1) {
      if (n < p.N) {
#pragma unroll
        for (int m = 0; m < M; ++m) p.y[(int64_t)m * p.N + n] = float_to_bf16_bits_rn(acc[m] * sc);
      }
    } else {
      const int my_slot = (rb == rb_first) ? 0 : 1;
      float* wsp = p.ws + ((int64_t)blockIdx.x * 2 + my_slot) * (kRows * kMaxTokens);
#pragma unroll
      for (int m = 0; m < M; ++m) __stcg(wsp + m * kRows + tid, acc[m]);
      __threadfence();
      named_bar_sync(1, kConsumerWarps * 32);
      const int64_t i_first = owner_of(seg_begin, p.W, p.G);
      const int64_t i_last = owner_of(seg_begin + T - 1, p.W, p.G);
      const int sf = (range_begin(i_first, p.W, p.G) / T == rb) ? 0 : 1;
      int* ctr = p.cnt + i_first * 2 + sf;
      if (tid == 0) {
        const int old = atomicAdd(ctr, 1);
        *s_flag = (old == (int)(i_last - i_first)) ? 1 : 0;
      }
      named_bar_sync(1, kConsumerWarps * 32);
      if (*s_flag) {
        __threadfence();
        float sum[M];
#pragma unroll
        for (int m = 0; m < M; ++m) sum[m] = 0.f;
        for (int64_t i = i_first; i <= i_last; ++i) {
          const int sl = (range_begin(i, p.W, p.G) / T == rb) ? 0 : 1;
          const float* src = p.ws + (i * 2 + sl) * (kRows * kMaxTokens);
#pragma unroll
          for (int m = 0; m < M; ++m) sum[m] += __ldcg(src + m * kRows + tid);
        }
        if (n < p.N) {
#pragma unroll
          for (int m = 0; m < M; ++m) p.y[(int64_t)m * p.N + n] = float_to_bf16_bits_rn(sum[m] * sc);
        }
        if (tid == 0) atomicExch(ctr, 0);
      }
      named_bar_sync(1, kConsumerWarps * 32);
    }
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] = 0.f;
  }
}

template <int M, int ES>
sp_status launch_one(const LinearParams& p, cudaStream_t stream, size_t smem) {
  auto kern = linear_cc_kernel<M, ES>;
  static bool configured[kMaxDevices] = {};  // the smem opt-in is set once per device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= kMaxDevices) return SP_ERR_UNSUPPORTED;
  if (!configured[dev]) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemOptIn) != cudaSuccess)
      return SP_ERR_CUDA;
    configured[dev] = true;
  }
  kern<<<p.G, kThreads, smem, stream>>>(p);
  return cudaGetLastError() == cudaSuccess ? SP_OK : SP_ERR_CUDA;
}

template <int ES>
sp_status dispatch_m(const LinearParams& p, cudaStream_t stream, size_t smem) {
  switch (p.M) {
    case 1: return launch_one<1, ES>(p, stream, smem);
    case 2: return launch_one<2, ES>(p, stream, smem);
    case 3: return launch_one<3, ES>(p, stream, smem);
    case 4: return launch_one<4, ES>(p, stream, smem);
    case 5: return launch_one<5, ES>(p, stream, smem);
    case 6: return launch_one<6, ES>(p, stream, smem);
    case 7: return launch_one<7, ES>(p, stream, smem);
    case 8: return launch_one<8, ES>(p, stream, smem);
    default: return SP_ERR_INVALID_ARG;
  }
}

int grid_cc(const sp_matrix* h) {
  const int64_t W = (int64_t)h->RB * h->T;
  static_assert(2 <= kMaxGridPerSm, "grid must fit the workspace counter region");
  return (int)std::min<int64_t>((int64_t)2 * h->num_sms, W);
}

}  // namespace

size_t workspace_bytes_cc(const sp_matrix* h, int64_t /*M*/) {
  const size_t G = (size_t)grid_cc(h);
  return ws_counter_bytes(h->num_sms) + 2 * G * kRows * kMaxTokens * sizeof(float);
}

sp_status launch_linear_cc(const sp_matrix* h, const uint16_t* x, int64_t M, uint16_t* y, void* ws, size_t ws_bytes,
                           cudaStream_t stream) {
  const size_t need = workspace_bytes_cc(h, M);
  if (!ws || ws_bytes < need) return SP_ERR_WORKSPACE;
  LinearParams p{};
  p.buf = h->d_buf;
  p.off = h->d_off;
  p.scale = h->d_scale;
  p.status = device_status_ptr();
  p.N = h->N;
  p.K = h->K;
  p.T = h->T;
  p.RB = h->RB;
  p.W = (int64_t)h->RB * h->T;
  p.G = grid_cc(h);
  p.cnt = reinterpret_cast<int*>(ws);
  p.ws = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(ws) + ws_counter_bytes(h->num_sms));
  p.timeout_ns = wait_timeout_ns();
  p.chunk_region = (uint32_t)((h->max_chunk + 127) / 128 * 128);
  for (int64_t m0 = 0; m0 < M; m0 += kMaxTokens) {
    const int Mt = (int)std::min<int64_t>(kMaxTokens, M - m0);
    p.M = Mt;
    p.x = x + m0 * h->K;
    p.y = y + m0 * h->N;
    p.slot_bytes = p.chunk_region + (uint32_t)Mt * 128u;
    // slots plus 2*slots mbarriers (<= 256 B) plus the flag must fit the budget
    int slots = (int)std::min<size_t>(16, (kSmemBudget - 256 - 16) / p.slot_bytes);
    if (slots < 2) return SP_ERR_UNSUPPORTED;
    p.slots = slots;
    const size_t smem = (size_t)slots * p.slot_bytes + 2 * (size_t)slots * 8 + 16;
    const sp_status st = h->esize == 2 ? dispatch_m<2>(p, stream, smem) : dispatch_m<1>(p, stream, smem);
    if (st != SP_OK) return st;
  }
  return SP_OK;
}

}  // namespace sp
