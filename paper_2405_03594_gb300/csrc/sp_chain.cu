// sp_chain.cu -- a chain of sparse linears (a decode step) in one persistent launch.
//
// y_k = epilogue_k(x_k . (W_k o Mask_k)^T) for k = 0, 1, ..., where x_k is (a view of)
// an earlier output: decode through the layers of a model, where every linear's
// compressed weight bytes stream from HBM once (Sec. 2.4.2: compressed submatrices move
// from global memory onto the chip and are expanded there; decode is bound by those
// bytes, Sec. 2.4, 3.4).  Launching one kernel per linear leaves every launch's tail idle
// on HBM; here the copies of the next linears' weights go out while the current linear's
// arithmetic finishes, and only the arithmetic of linear k waits for linear k-1.
//
// Work split: one CTA per SM.  A unit of work is one 32-row quarter of a 128-row block over
// the whole K range, so each output row is summed inside one CTA: no split-K partials
// leave the SM and no fix-up runs between CTAs.  CTA i takes units i, i + G, i + 2G, ...
// of every linear; its NW warps (16 to 32, chain_warps below) take the unit's K-tiles
// round-robin (warp w the CTA's items n with n % NW == w) and add their partial sums in
// shared memory in warp order (deterministic).  Per item (unit, K-tile) a warp:
//   - has issued, D items earlier, two bulk copies into one of its own ring slots: the
//     quarter's 32 row masks (256 bytes) and the span of chunk bytes holding its kept
//     values (located by the per-chunk quarter index built at compression);
//   - lane r <-> row 32q + r: popc prefix for the row's first value, two-chain bit walk,
//     x by shuffle (x loaded from global memory one item ahead), FP32 accumulation.
// Dependencies: when a CTA has written its rows of linear k it adds 1 to done[k]
// (release, GPU scope); a CTA starts the arithmetic of linear k+1 once done[k] == G
// (acquire).  Weight copies never wait.
// Epilogues: store: y = bf16(s * acc); residual: y = bf16((y + bf16(s * acc)) + r) in
// place; pair product (rows 2j, 2j+1): y[:, j] = bf16(bf16(s * acc_2j) * bf16(s * acc_2j+1)).
// The last CTA to finish clears the counters, so each call leaves the workspace ready for
// the next one.
#include <algorithm>

#include "../../include/sp_stack.h"
#include "sp_cc_common.cuh"

namespace sp {
namespace {

using namespace cc;

constexpr int kChainMaxOps = 160;  // linears per launch (they travel in the kernel parameters)
constexpr int kChainMaxM = 4;      // batch rows
// Warps per CTA (every warp walks chunks and issues its own copies): 32 at M = 1 (64
// registers, no spills; measured on GB300, the 32-layer step at 70%: 2.386 -> 2.339 ms
// against 24 warps), 24 while the batch loop fits 85 registers (M <= 3), else 16.
__host__ __device__ constexpr int chain_warps(int m) { return m == 1 ? 32 : m <= 3 ? 24 : 16; }
constexpr int kMaxDevices = 64;

struct ChainOpDev {
  const uint8_t* buf;
  const uint64_t* off;
  const uint64_t* qidx;  // quarter index: kept entries before rows 32, 64, 96 and in all rows
  const float* scale;    // INT8 only
  const uint16_t* x;     // bf16 [M, ldx]
  uint16_t* y;           // bf16 [M, ldy]
  const uint16_t* r;     // residual vector [N] (SP_EPI_RESIDUAL)
  int32_t N, K, T, RB;
  int32_t ldx, ldy;
  int32_t epi, esize;
};

struct ChainParams {
  int32_t n_ops, M, G, depth;  // depth D: ring slots per warp
  uint32_t slot_bytes, comb_off;
  int* done;    // [kChainMaxOps] per-linear completion counts, then the exit count
  int* status;
  uint64_t timeout_ns;
  ChainOpDev ops[kChainMaxOps];
};

// Workspace: the completion counters and the exit count.
constexpr size_t kChainWsBytes = ((kChainMaxOps + 1) * sizeof(int) + 255) / 256 * 256;

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_relaxed(const int* p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// x[m, 64t + lane] and x[m, 64t + 32 + lane] of linear `op`, two batch rows per register,
// by coherent (L2) loads: x was written by other CTAs during this launch.
template <int M>
__device__ __forceinline__ void load_x_global(const ChainOpDev& op, int t, int lane, uint32_t (&XL)[(M + 1) / 2],
                                              uint32_t (&XH)[(M + 1) / 2]) {
  const int c0 = kTileK * t + lane, c1 = c0 + 32;
  const bool v0 = c0 < op.K, v1 = c1 < op.K;
#pragma unroll
  for (int q = 0; q < (M + 1) / 2; ++q) {
    const unsigned short* r0 = op.x + (size_t)(2 * q) * op.ldx;
    uint32_t a0 = v0 ? __ldcg(r0 + c0) : 0u, b0 = v1 ? __ldcg(r0 + c1) : 0u, a1 = 0u, b1 = 0u;
    if (2 * q + 1 < M) {
      const unsigned short* r1 = r0 + op.ldx;
      a1 = v0 ? __ldcg(r1 + c0) : 0u;
      b1 = v1 ? __ldcg(r1 + c1) : 0u;
    }
    XL[q] = a0 | (a1 << 16);
    XH[q] = b0 | (b1 << 16);
  }
}

// Output row n of linear `op` from its FP32 sums v.  All 32 lanes of the warp call this
// together (the pair product exchanges sums between neighbouring lanes).
template <int M, int ES>
__device__ __forceinline__ void chain_write(const ChainOpDev& op, int64_t n, const float (&v)[M]) {
  const bool in = n < op.N;
  const float sc = (ES == 1 && in) ? __ldg(op.scale + n) : 1.f;
  if (op.epi == SP_EPI_STORE) {
    if (in) {
#pragma unroll
      for (int m = 0; m < M; ++m) op.y[(int64_t)m * op.ldy + n] = float_to_bf16_bits_rn(v[m] * sc);
    }
  } else if (op.epi == SP_EPI_RESIDUAL) {
    if (in) {
      const float rv = bf16_bits_to_float(__ldg(op.r + n));
#pragma unroll
      for (int m = 0; m < M; ++m) {
        uint16_t* yp = op.y + (int64_t)m * op.ldy + n;
        const float a = bf16_bits_to_float(float_to_bf16_bits_rn(v[m] * sc));
        const float h = bf16_bits_to_float(__ldcg(reinterpret_cast<const unsigned short*>(yp)));
        *yp = float_to_bf16_bits_rn((h + a) + rv);
      }
    }
  } else {  // SP_EPI_PAIR_PRODUCT
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const uint32_t g = in ? float_to_bf16_bits_rn(v[m] * sc) : 0u;
      const uint32_t u = __shfl_xor_sync(0xffffffffu, g, 1);
      if (in && (n & 1) == 0)
        op.y[(int64_t)m * op.ldy + (n >> 1)] = float_to_bf16_bits_rn(bf16_bits_to_float(g) * bf16_bits_to_float(u));
    }
  }
}

// ---------------------------------------------------------------- work walk
// The items of linear k are (unit u, K-tile t) with unit u = 4*rb + q (row block rb,
// quarter q), in unit-major order over the units of this CTA (u = blockIdx.x + j*G).  The
// CTA's n-th item overall (counting across linears) belongs to warp n % NW (NW warps), which
// owns ring slots w, w + NW, ..., and takes its m-th item into slot w + NW*(m % D).
struct OpShape {
  int32_t T, U, J;  // K-tiles, units, units of this CTA
  __device__ __forceinline__ void load(const ChainParams& p, int k) {
    T = p.ops[k].T;
    U = 4 * p.ops[k].RB;
    J = (int)blockIdx.x < U ? (U - 1 - (int)blockIdx.x) / p.G + 1 : 0;
  }
};
// first K-tile of unit j that warp w owns, given the CTA's item count n0 before linear k
template <int NW>
__device__ __forceinline__ int first_t(int w, int64_t n0, int j, int T) {
  const int r = (int)(((int64_t)w - n0 - (int64_t)j * T) % NW);
  return r < 0 ? r + NW : r;
}

// Walks warp w's items in order across linears (the issue side runs ahead of the math).
template <int NW>
struct ItemWalk {
  int k, j, t;
  int64_t n0;  // CTA items before linear k
  OpShape sh;
  __device__ __forceinline__ void settle(const ChainParams& p, int w) {
    // move to the first valid item at or after (k, j, t)
    while (k < p.n_ops) {
      if (j < sh.J) {
        if (t < sh.T) return;
        ++j;
        if (j < sh.J) t = first_t<NW>(w, n0, j, sh.T);
        continue;
      }
      n0 += (int64_t)sh.J * sh.T;
      if (++k < p.n_ops) {
        sh.load(p, k);
        j = 0;
        t = sh.J > 0 ? first_t<NW>(w, n0, 0, sh.T) : 0;
      }
    }
  }
  __device__ __forceinline__ void start(const ChainParams& p, int w) {
    k = 0;
    n0 = 0;
    sh.load(p, 0);
    j = 0;
    t = sh.J > 0 ? first_t<NW>(w, 0, 0, sh.T) : 0;
    settle(p, w);
  }
  __device__ __forceinline__ void next(const ChainParams& p, int w) {
    t += NW;
    settle(p, w);
  }
  __device__ __forceinline__ bool valid(const ChainParams& p) const { return k < p.n_ops; }
};

// Chunk number and quarter of the walk's current item.
template <class Walk>
__device__ __forceinline__ void item_chunk(const ChainParams& p, const Walk& it, int64_t* c, int* q) {
  const int u = (int)blockIdx.x + it.j * p.G;
  *c = (int64_t)(u >> 2) * it.sh.T + it.t;
  *q = u & 3;
}

// Offsets of the walk's current item (lane 0 loads them one issue ahead of their use).
struct ItemOffsets {
  uint64_t off, qi;
  template <class Walk>
  __device__ __forceinline__ void load(const ChainParams& p, const Walk& it) {
    int64_t c;
    int q;
    item_chunk(p, it, &c, &q);
    off = __ldg(p.ops[it.k].off + c);
    qi = __ldg(p.ops[it.k].qidx + c);
  }
};

// Issue the copies of one item into slot `s` (lane 0): the quarter's 32 row masks (256
// bytes) and the 16-byte-aligned span of chunk bytes that holds its kept values.  The offset
// of the quarter's first value inside that span goes to voff[s].
template <class Walk>
__device__ __forceinline__ void issue_item(const ChainParams& p, const Walk& it, const ItemOffsets& io,
                                           uint8_t* slot, uint64_t* full, volatile uint32_t* voff, uint64_t pol) {
  const ChainOpDev& op = p.ops[it.k];
  int64_t c;
  int q;
  item_chunk(p, it, &c, &q);
  const uint32_t s0 = q == 0 ? 0u : (uint32_t)(io.qi >> (16 * (q - 1))) & 0xffffu;
  const uint32_t s1 = (uint32_t)(io.qi >> (16 * q)) & 0xffffu;
  const uint32_t b0 = kMaskBytes + s0 * (uint32_t)op.esize, b1 = kMaskBytes + s1 * (uint32_t)op.esize;
  const uint32_t a0 = b0 & ~15u, a1 = (b1 + 15u) & ~15u;
  *voff = b0 - a0;
  mbar_arrive_expect_tx(full, 256u + (a1 - a0));
  bulk_g2s_hint(slot, op.buf + io.off + 256u * (uint32_t)q, 256u, full, pol);
  if (a1 > a0) bulk_g2s_hint(slot + 256, op.buf + io.off + a0, a1 - a0, full, pol);
}

// Shared-memory control of the asynchronous unit ends: flushed[b] counts the warps that
// deposited their partials in combine buffer b; ready[b] is the CTA unit count that may use
// buffer b next.
struct UnitCtl {
  int flushed[2];
  int ready[2];
};

template <int M, int ES>
__device__ __forceinline__ void chain_warp(const ChainParams& p, uint8_t* smem, uint64_t* full,
                                           volatile uint32_t* voff, float* comb, volatile UnitCtl* ctl,
                                           volatile int* s_flag, int warp, int lane) {
  constexpr int MP = (M + 1) / 2;
  constexpr int NW = chain_warps(M);
  const int D = p.depth;
  const uint64_t pol = policy_evict_first();
  auto slot_of = [&](int d) { return warp + NW * d; };
  // ---- issue side: the first D items
  ItemWalk<NW> iw;
  iw.start(p, warp);
  ItemOffsets io;
  if (lane == 0 && iw.valid(p)) io.load(p, iw);
  int issued = 0;  // items of this warp whose copies went out
  for (; issued < D && iw.valid(p); ++issued) {
    const int s = slot_of(issued);
    if (lane == 0) issue_item(p, iw, io, smem + (size_t)s * p.slot_bytes, &full[s], &voff[s], pol);
    iw.next(p, warp);
    if (lane == 0 && iw.valid(p)) io.load(p, iw);
  }
  // ---- math side
  bool dead = false;
  int m = 0;       // items of this warp walked so far
  int dcur = 0;    // ring position of item m (m % D) and its phase parity ((m / D) & 1)
  uint32_t phase = 0;
  int waited = 0;  // items whose copies this warp has seen land
  int ucnt = 0;    // units of this CTA finished so far (all linears)
  int64_t n0 = 0;
  for (int k = 0; k < p.n_ops; ++k) {
    const ChainOpDev& op = p.ops[k];
    OpShape sh;
    sh.load(p, k);
    if (sh.J > 0) {
      if (k > 0) {
        // linear k-1 complete on every CTA: its output (this linear's x) is in memory
        if (warp == 0 && lane == 0 && !s_flag[1]) {
          const int* dp = p.done + (k - 1);
          if (ld_acquire(dp) < p.G) {
            const uint64_t t0 = global_ns();
            while (ld_acquire(dp) < p.G) {
              __nanosleep(32);
              if (global_ns() - t0 > p.timeout_ns || ld_relaxed(p.status) != kStatusOk) {
                set_status(p.status, kStatusTimeout);
                s_flag[1] = 1;
                break;
              }
            }
          }
        }
        named_bar_sync(1, NW * 32);
      }
      dead = dead || __any_sync(0xffffffffu, s_flag[1] != 0);
      uint32_t XL[MP], XH[MP], XLn[MP], XHn[MP];
      // this warp's first item of the linear, for the x prefetch
      int jx = 0, tx = first_t<NW>(warp, n0, 0, sh.T);
      while (jx < sh.J && tx >= sh.T) {
        ++jx;
        if (jx < sh.J) tx = first_t<NW>(warp, n0, jx, sh.T);
      }
      if (jx < sh.J) load_x_global<M>(op, tx, lane, XL, XH);
      for (int j = 0; j < sh.J; ++j) {
        const int u = (int)blockIdx.x + j * p.G;
        float acc[M];
#pragma unroll
        for (int mm = 0; mm < M; ++mm) acc[mm] = 0.f;
        for (int t = first_t<NW>(warp, n0, j, sh.T); t < sh.T; t += NW) {
          // x of this warp's next item in the linear (the same unit or a later one)
          {
            int jn = j, tn = t + NW;
            while (jn < sh.J && tn >= sh.T) {
              ++jn;
              if (jn < sh.J) tn = first_t<NW>(warp, n0, jn, sh.T);
            }
            if (jn < sh.J) load_x_global<M>(op, tn, lane, XLn, XHn);
          }
          const int s = slot_of(dcur);
          if (!dead) {
            const bool ok = __all_sync(0xffffffffu, mbar_wait_sleep(&full[s], phase, p.timeout_ns));
            if (!ok) {
              dead = true;
              set_status(p.status, kStatusTimeout);
              s_flag[1] = 1;
            } else {
              ++waited;
            }
          }
          if (!dead) {
            const uint8_t* slot = smem + (size_t)s * p.slot_bytes;
            const uint64_t mk = reinterpret_cast<const uint64_t*>(slot)[lane];
            const uint32_t lo = (uint32_t)mk, hi = (uint32_t)(mk >> 32);
            const int plo = __popc(lo), pc = plo + __popc(hi);
            int incl = pc;
#pragma unroll
            for (int dd = 1; dd < 32; dd <<= 1) {
              const int v = __shfl_up_sync(0xffffffffu, incl, dd);
              if (lane >= dd) incl += v;
            }
            const uint32_t vo = voff[s];
            row_dot<M, ES>(lo, hi, plo, pc, incl - pc, slot + 256 + vo, XL, XH, acc);
          }
          __syncwarp();
          ++m;
          if (++dcur == D) {
            dcur = 0;
            phase ^= 1u;
          }
          // the slot is free again: refill it with this warp's item D positions ahead
          if (iw.valid(p) && !dead) {
            if (lane == 0) issue_item(p, iw, io, smem + (size_t)s * p.slot_bytes, &full[s], &voff[s], pol);
            iw.next(p, warp);
            if (lane == 0 && iw.valid(p)) io.load(p, iw);
            ++issued;
          }
#pragma unroll
          for (int q = 0; q < MP; ++q) {
            XL[q] = XLn[q];
            XH[q] = XHn[q];
          }
        }
        // unit end: the warps' partial sums for rows 32q + lane go to combine buffer b; the
        // last warp to deposit adds them in warp order and writes the rows, while the others
        // go on with their next unit (no barrier).  Buffer b serves units ucnt, ucnt + 2, ...
        const int b = (int)(ucnt & 1);
        if (ctl->ready[b] != ucnt) {
          const uint64_t t0 = global_ns();
          while (ctl->ready[b] != ucnt) {
            __nanosleep(32);
            if (global_ns() - t0 > p.timeout_ns) {
              set_status(p.status, kStatusTimeout);
              s_flag[1] = 1;
              break;
            }
          }
        }
        float* cb = comb + (size_t)b * NW * M * 32;
#pragma unroll
        for (int mm = 0; mm < M; ++mm) cb[(warp * M + mm) * 32 + lane] = acc[mm];
        __syncwarp();
        int last = 0;
        if (lane == 0) {
          __threadfence_block();
          last = atomicAdd(const_cast<int*>(&ctl->flushed[b]), 1) == NW - 1 ? 1 : 0;
        }
        if (__shfl_sync(0xffffffffu, last, 0)) {
          __threadfence_block();
          float sum[M];
#pragma unroll
          for (int mm = 0; mm < M; ++mm) {
            float a = cb[mm * 32 + lane];
            for (int w = 1; w < NW; ++w) a += cb[(w * M + mm) * 32 + lane];
            sum[mm] = a;
          }
          chain_write<M, ES>(op, (int64_t)(u >> 2) * kRows + 32 * (u & 3) + lane, sum);
          __syncwarp();
          if (lane == 0) {
            ctl->flushed[b] = 0;
            __threadfence_block();
            ctl->ready[b] = ucnt + 2;
          }
        }
        ++ucnt;
      }
      // this CTA is done with linear k once every warp has deposited its last partial and the
      // last unit's rows are written (the writer arrives here after writing them)
      named_bar_sync(1, NW * 32);
    }
    if (warp == 0 && lane == 0) red_release_add(p.done + k, 1);
    n0 += (int64_t)sh.J * sh.T;
  }
  // copies still in flight (only if a wait gave up) must land before the CTA exits
  if (lane == 0) {
    for (int i = waited; i < issued; ++i) mbar_wait(&full[slot_of(i % D)], (uint32_t)((i / D) & 1), p.timeout_ns);
  }
}

template <int M, int ES>
__global__ void __launch_bounds__(chain_warps(M) * 32, 1) chain_kernel(const __grid_constant__ ChainParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int NW = chain_warps(M);
  const int S = NW * p.depth;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)S * p.slot_bytes);
  volatile uint32_t* voff = reinterpret_cast<volatile uint32_t*>(full + S);
  float* comb = reinterpret_cast<float*>(smem + p.comb_off);
  volatile UnitCtl* ctl = reinterpret_cast<volatile UnitCtl*>(comb + 2 * NW * M * 32);
  volatile int* s_flag = reinterpret_cast<volatile int*>(ctl + 1);  // [1] a wait gave up
  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(&full[s], 1);
    s_flag[0] = 0;
    s_flag[1] = 0;
    ctl->flushed[0] = ctl->flushed[1] = 0;
    ctl->ready[0] = 0;
    ctl->ready[1] = 1;
    fence_barrier_init();
  }
  __syncthreads();
  chain_warp<M, ES>(p, smem, full, voff, comb, ctl, s_flag, warp, lane);
  __syncthreads();
  if (tid == 0) {
    // the last CTA out clears the completion counters for the next call (every other CTA
    // has finished all its waits on them)
    __threadfence();
    int* exit_cnt = p.done + kChainMaxOps;
    if (atomicAdd(exit_cnt, 1) == p.G - 1) {
      __threadfence();
      for (int k = 0; k < p.n_ops; ++k) atomicExch(p.done + k, 0);
      atomicExch(exit_cnt, 0);
    }
  }
}

template <int M, int ES>
sp_status launch_chain(ChainParams& p, cudaStream_t stream, size_t smem, int dev) {
  auto kern = chain_kernel<M, ES>;
  static size_t configured[kMaxDevices] = {};
  if (configured[dev] < smem) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
      cudaGetLastError();
      return SP_ERR_CUDA;
    }
    configured[dev] = smem;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, chain_warps(M) * 32, smem) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  int num_sms = 0;
  cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev);
  if (per_sm < 1 || num_sms < 1) return SP_ERR_UNSUPPORTED;
  p.G = num_sms;  // one CTA per SM
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.G);
  cfg.blockDim = dim3(chain_warps(M) * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident: they wait on one another
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, kern, p) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  return SP_OK;
}

template <int ES>
sp_status dispatch_chain(ChainParams& p, cudaStream_t stream, size_t smem, int dev) {
  switch (p.M) {
    case 1: return launch_chain<1, ES>(p, stream, smem, dev);
    case 2: return launch_chain<2, ES>(p, stream, smem, dev);
    case 3: return launch_chain<3, ES>(p, stream, smem, dev);
    case 4: return launch_chain<4, ES>(p, stream, smem, dev);
    default: return SP_ERR_UNSUPPORTED;
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned2(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 1u) == 0; }

}  // namespace
}  // namespace sp

using namespace sp;

extern "C" {

sp_status sp_chain_workspace_size(int64_t m, size_t* bytes) {
  if (!bytes || m < 0) return SP_ERR_INVALID_ARG;
  *bytes = m == 0 ? 0 : kChainWsBytes;
  return SP_OK;
}

sp_status sp_chain_run(const sp_chain_op* ops, int32_t n_ops, int64_t m, void* workspace_dev, size_t workspace_bytes,
                       void* stream) {
  if (!ops || n_ops < 0 || m < 0) return SP_ERR_INVALID_ARG;
  if (m == 0 || n_ops == 0) return SP_OK;
  if (m > kChainMaxM) return SP_ERR_UNSUPPORTED;
  int dev = -1, smem_optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices ||
      cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  if (!workspace_dev || workspace_bytes < kChainWsBytes) return SP_ERR_WORKSPACE;
  if (!aligned16(workspace_dev)) return SP_ERR_ALIGNMENT;
  int esize = 0;
  for (int32_t k = 0; k < n_ops; ++k) {
    const sp_chain_op& o = ops[k];
    const sp_matrix* h = o.w;
    if (!h || h->magic != SP_MAGIC) return SP_ERR_BAD_HANDLE;
    if (h->device != dev) return SP_ERR_INVALID_ARG;
    if (!o.x || !o.y || (o.epilogue == SP_EPI_RESIDUAL && !o.r)) return SP_ERR_INVALID_ARG;
    if (o.epilogue != SP_EPI_STORE && o.epilogue != SP_EPI_RESIDUAL && o.epilogue != SP_EPI_PAIR_PRODUCT)
      return SP_ERR_INVALID_ARG;
    const int64_t ny = o.epilogue == SP_EPI_PAIR_PRODUCT ? h->N / 2 : h->N;
    if (o.ldx < h->K || o.ldy < ny || (o.epilogue == SP_EPI_PAIR_PRODUCT && h->N % 2 != 0))
      return SP_ERR_INVALID_ARG;
    if (o.ldx > INT32_MAX || o.ldy > INT32_MAX || h->N > INT32_MAX || h->K > INT32_MAX ||
        (int64_t)4 * h->RB > INT32_MAX)
      return SP_ERR_UNSUPPORTED;
    if (!aligned2(o.x) || !aligned2(o.y) || (o.r && !aligned2(o.r))) return SP_ERR_ALIGNMENT;
    if (k == 0) esize = h->esize;
    if (h->esize != esize) return SP_ERR_UNSUPPORTED;  // one value type per chain
  }
  int* status = device_status_ptr();
  if (!status) return SP_ERR_CUDA;
  ChainParams p;  // copied into the launch's parameters
  for (int32_t k0 = 0; k0 < n_ops; k0 += kChainMaxOps) {
    const int32_t nk = std::min<int32_t>(kChainMaxOps, n_ops - k0);
    p = ChainParams{};
    p.n_ops = nk;
    p.M = (int32_t)m;
    p.done = static_cast<int*>(workspace_dev);
    p.status = status;
    p.timeout_ns = wait_timeout_ns();
    uint32_t max_quarter = 1;
    for (int32_t k = 0; k < nk; ++k) {
      const sp_chain_op& o = ops[k0 + k];
      const sp_matrix* h = o.w;
      ChainOpDev& d = p.ops[k];
      d.buf = h->d_buf;
      d.off = h->d_off;
      d.qidx = h->d_qidx;
      d.scale = h->d_scale;
      d.x = static_cast<const uint16_t*>(o.x);
      d.y = static_cast<uint16_t*>(o.y);
      d.r = static_cast<const uint16_t*>(o.r);
      d.N = (int32_t)h->N;
      d.K = (int32_t)h->K;
      d.T = h->T;
      d.RB = h->RB;
      d.ldx = (int32_t)o.ldx;
      d.ldy = (int32_t)o.ldy;
      d.epi = o.epilogue;
      d.esize = h->esize;
      max_quarter = std::max(max_quarter, h->max_quarter);
    }
    // A slot holds a quarter's 256 bytes of masks and the 16-byte-aligned span of its values
    // (at most its value bytes + 30, rounded to 16).
    p.slot_bytes = 256u + ((uint32_t)esize * max_quarter + 15u) / 16u * 16u + 16u;
    const int nw = chain_warps((int)m);
    const size_t comb = (size_t)2 * nw * m * 32 * sizeof(float);
    const size_t budget = (size_t)smem_optin - 1024;
    const size_t per_depth = (size_t)nw * (p.slot_bytes + sizeof(uint64_t) + sizeof(uint32_t));
    if (budget < comb + 32 + 2 * per_depth) return SP_ERR_UNSUPPORTED;
    p.depth = (int)std::min<size_t>(16, (budget - comb - 32) / per_depth);
    const size_t S = (size_t)nw * p.depth;
    p.comb_off = (uint32_t)((S * (p.slot_bytes + sizeof(uint64_t) + sizeof(uint32_t)) + 15) / 16 * 16);
    const size_t smem = p.comb_off + comb + 32;
    const sp_status st = esize == 2 ? dispatch_chain<2>(p, (cudaStream_t)stream, smem, dev)
                                    : dispatch_chain<1>(p, (cudaStream_t)stream, smem, dev);
    if (st != SP_OK) return st;
  }
  return SP_OK;
}

}  // extern "C"
