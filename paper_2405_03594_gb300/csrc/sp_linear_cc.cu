// sp_linear_cc.cu -- decode-batch sparse linear on the CUDA cores.
//
// y[m, n] = sum_k x[m, k] * W[n, k] over the kept entries, read straight from the
// compressed chunks (Sec. 2.4.2: the compressed submatrices move from global
// memory onto the chip and are expanded there by their bitmask; decode is bound
// by those bytes, Sec. 2.4, 3.4).
//
// Launch: each row block split over the S CTAs of a thread-block cluster (partials summed
// over distributed shared memory), or -- when not even two CTAs per row block fit -- G
// CTAs each owning a contiguous run of chunks in storage order (stream-K), so every CTA
// streams one linear byte range.  Four CTAs per SM, six for one-row warp-per-chunk
// cluster launches (cluster_cc and select_cc below).
//   warp 4, lane 0   producer: one cp.async.bulk per chunk (+ one copy of
//                    x[m, 64t : 64t+64) per batch row) into a ring of `slots`
//                    shared-memory slots, each guarded by a full/empty mbarrier
//                    pair; weight bytes carry an L2 evict-first hint.
//   warps 0-3        consumers, thread r <-> row r of the chunk: its first value is
//                    found by a popc prefix sum over the chunk's masks (warp scan plus
//                    the other warps' redux sums); it walks its set bits (two
//                    independent chains: columns 0-31 and 32-63), gathers
//                    x[m, 64t+j] from lane j%32 by shuffle (two batch rows per
//                    register), and accumulates with the FP32-accumulating bf16 FMA.
//                    At a row-block end the 128 rows are written (bf16, RNE, through
//                    the launch's output epilogue), or -- when the row block is shared
//                    with other CTAs outside a cluster -- stored as an FP32 partial and
//                    summed in CTA order by the last CTA to arrive (deterministic
//                    split-K).  The warp-per-chunk kernel (M <= 4) is described at its
//                    definition below.
#include <algorithm>

#include "../../include/sp_stack.h"
#include "sp_cc_common.cuh"

namespace sp {
namespace {

using namespace cc;

constexpr int kConsumerWarps = 4;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kMaxDevices = 64;
constexpr int kCtasPerSm = 4;
constexpr size_t kSmemBudget = 53 * 1024;  // ring slots per CTA; four CTAs share one SM
constexpr size_t kSmemOptIn = 54 * 1024;
// Warp-per-chunk cluster launches at M = 1 run six CTAs per SM (64 registers, no spills;
// 24 consumer warps per SM instead of 16 to cover the walk's latencies) when four ring
// slots of the matrix's largest chunk fit the smaller budget; other launches spill at 64
// registers and keep four.
constexpr int kCtasPerSmM1 = 6;
constexpr size_t kSmemBudgetM1 = 37 * 1024;
// Where four slots of the largest chunk do not fit that budget (50 % sparsity: ~9.2 KB
// chunks), one-row cluster launches run five CTAs per SM (72 registers, no spills; 44 KB).
constexpr int kCtasPerSmM1b = 5;
constexpr size_t kSmemBudgetM1b = 44 * 1024;

// CTA's work items [w0, w1): a contiguous run of chunks (stream-K), or -- in cluster
// mode -- K-tiles [r*T/S, (r+1)*T/S) of the row block of its cluster (r = its rank).
__device__ __forceinline__ void cta_range(const LinearParams& p, bool clustered, int64_t* w0, int64_t* w1,
                                          uint32_t* crank) {
  if (clustered) {
    const int64_t seg = blockIdx.x / p.cluster;
    *crank = cluster_rank();
    *w0 = seg * p.T + (int64_t)*crank * p.T / p.cluster;
    *w1 = seg * p.T + (int64_t)(*crank + 1) * p.T / p.cluster;
  } else {
    *crank = 0;
    *w0 = range_begin(blockIdx.x, p.W, p.G);
    *w1 = range_begin(blockIdx.x + 1, p.W, p.G);
  }
}

// Producer warp: one cp.async.bulk per chunk (evict-first L2 hint) plus one copy of
// x[m, 64t : 64t+64) per batch row into ring slot n % slots, in item order.  The whole
// warp walks the chunk list (it shares the offset window); lane 0 issues.  Weight bytes
// do not depend on the previous kernel in the stream: the first ring fill is issued
// before griddepcontrol.wait; every x copy comes after it.  EARLY: release the next
// launch in the stream as soon as the dependency is met (the six-CTA M = 1 launches);
// otherwise the release comes with the CTA's exit.  Measured on GB300 (32-layer decode
// step, 70%): releasing at exit made the four-CTA launches' steps 6-7% faster at M = 4
// and 8 (their CTAs no longer land in whatever slots the previous launch's tail leaves),
// while at M = 1 early release is what lets six-CTA launches overlap.
// tag[s] = n records that slot s has been claimed for item n (written once the slot's
// previous item has been consumed), for consumers that do not read every item.
template <int M, bool EARLY = true>
__device__ __forceinline__ void produce(const LinearParams& p, uint8_t* smem, uint64_t* full, uint64_t* empty,
                                        volatile int* tag, int64_t w0, int64_t w1, int lane) {
  const int T = p.T;
  const int slots = p.slots;
  const uint64_t pol = policy_evict_first();
  OffsetWindow ow;
  ow.init(p.off, p.W + 1, w0);
  const int64_t n_pre = imin64((int64_t)slots, w1 - w0);
  {
    int t = (int)(w0 % T);
    for (int64_t i = 0; i < n_pre; ++i) {
      uint64_t o0, o1;
      ow.at(w0 + i, &o0, &o1);
      if (lane == 0) {
        const uint32_t bytes = (uint32_t)(o1 - o0);
        const int valid = (int)imin64((int64_t)kTileK, p.K - (int64_t)kTileK * t);
        tag[i] = (int)i;
        mbar_arrive_expect_tx(&full[i], bytes + (uint32_t)M * (uint32_t)valid * 2u);
        bulk_g2s_hint(smem + (size_t)i * p.slot_bytes, p.buf + o0, bytes, &full[i], pol);
      }
      if (++t == T) t = 0;
    }
  }
  pdl_wait();
  if constexpr (EARLY) pdl_launch_dependents();
  int s = 0;
  uint32_t ph = 0;
  int t = (int)(w0 % T);
  int64_t n_issued = 0;
  bool failed = false;
  for (int64_t w = w0; w < w1 && !failed; ++w, ++n_issued) {
    const int valid = (int)imin64((int64_t)kTileK, p.K - (int64_t)kTileK * t);
    const uint32_t xb = (uint32_t)valid * 2u;
    uint8_t* slot = smem + (size_t)s * p.slot_bytes;
    if (n_issued >= n_pre) {
      uint64_t o0, o1;
      ow.at(w, &o0, &o1);
      if (lane == 0) {
        if (!mbar_wait(&empty[s], ph ^ 1u, p.timeout_ns)) {
          set_status(p.status, kStatusTimeout);
          failed = true;
        } else {
          const uint32_t bytes = (uint32_t)(o1 - o0);
          tag[s] = (int)n_issued;
          mbar_arrive_expect_tx(&full[s], bytes + (uint32_t)M * xb);
          bulk_g2s_hint(slot, p.buf + o0, bytes, &full[s], pol);
        }
      }
      failed = __shfl_sync(0xffffffffu, failed, 0);
      if (failed) break;
    }
    if (lane == 0) {
#pragma unroll
      for (int m = 0; m < M; ++m)
        bulk_g2s(slot + p.chunk_region + m * 128, p.x + (int64_t)m * p.K + (int64_t)kTileK * t, xb, &full[s]);
    }
    if (++t == T) t = 0;
    if (++s == slots) {
      s = 0;
      ph ^= 1u;
    }
  }
}

// End of row block rb for consumer thread tid <-> output row rb*128 + tid, holding this
// CTA's FP32 sums `acc` over the row block's K-tiles it covered.
//  cluster mode: each CTA leaves its partial in its own shared memory; after a cluster
//    barrier rank 0 adds the other ranks' partials in rank order (distributed shared
//    memory) and writes y; a second barrier keeps every partial alive until then.
//  stream-K: a CTA that covered the whole row block (`complete`) writes y; otherwise it
//    stores its partial in workspace slot `my_slot` (0 = its first row block, 1 = its
//    last), and the last of the row block's CTAs to arrive sums the partials in CTA
//    order (deterministic) and writes y.
// All consumer threads (kConsumerWarps warps) call this together.
// Output of row n for the batch rows from its FP32 sums v (INT8: times the row's scale sc)
// through the launch's epilogue (the definitions of sp_chain_epilogue): store; residual,
// y = bf16((y + bf16(v sc)) + r[n]) in place; pair product of rows 2j and 2j+1 into y [m, N/2].
// All 32 lanes of a warp call it together with consecutive rows (the pair product takes the
// odd row's value from the neighbouring lane); rows past N write nothing.
template <int M>
__device__ __forceinline__ void write_row(const LinearParams& p, int64_t n, const float (&v)[M], float sc) {
  const bool in = n < p.N;
  if (p.epi == SP_EPI_PAIR_PRODUCT) {
    const int64_t ldy = p.N >> 1;
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const uint32_t g = in ? float_to_bf16_bits_rn(v[m] * sc) : 0u;
      const uint32_t u = __shfl_xor_sync(0xffffffffu, g, 1);
      if (in && (n & 1) == 0)
        p.y[(int64_t)m * ldy + (n >> 1)] = float_to_bf16_bits_rn(bf16_bits_to_float(g) * bf16_bits_to_float(u));
    }
  } else if (in) {
    if (p.epi == SP_EPI_RESIDUAL) {
      const float rv = bf16_bits_to_float(p.r[n]);
#pragma unroll
      for (int m = 0; m < M; ++m) {
        uint16_t* yp = p.y + (int64_t)m * p.N + n;
        const float a = bf16_bits_to_float(float_to_bf16_bits_rn(v[m] * sc));
        *yp = float_to_bf16_bits_rn((bf16_bits_to_float(__ldcg(reinterpret_cast<const unsigned short*>(yp))) + a) + rv);
      }
    } else {
#pragma unroll
      for (int m = 0; m < M; ++m) p.y[(int64_t)m * p.N + n] = float_to_bf16_bits_rn(v[m] * sc);
    }
  }
}

template <int M, int ES, bool CL>
__device__ __forceinline__ void row_block_end(const LinearParams& p, uint8_t* smem, volatile int* s_flag,
                                              const float (&acc)[M], int64_t rb, bool complete, int my_slot,
                                              uint32_t crank, int tid) {
  const int T = p.T;
  const int64_t seg_begin = rb * T;
  const int64_t n = rb * kRows + tid;
  const float sc = (ES == 1 && n < p.N) ? p.scale[n] : 1.f;
  if constexpr (CL) {
    float* part = reinterpret_cast<float*>(smem + p.part_off);
#pragma unroll
    for (int m = 0; m < M; ++m) part[m * kRows + tid] = acc[m];
    cluster_sync_all();
    if (crank == 0) {
      float sum[M];
#pragma unroll
      for (int m = 0; m < M; ++m) sum[m] = acc[m];
      const uint32_t base = smem_u32(part) + 4u * (uint32_t)tid;
      // the other ranks' partials, kR ranks' loads in flight at a time; the adds stay in
      // rank order
      constexpr int kR = M <= 2 ? 4 : 2;
      for (int r0 = 1; r0 < p.cluster; r0 += kR) {
        float v[kR][M];
#pragma unroll
        for (int u = 0; u < kR; ++u)
          if (r0 + u < p.cluster) {
            const uint32_t rb_addr = cluster_map(base, (uint32_t)(r0 + u));
#pragma unroll
            for (int m = 0; m < M; ++m) v[u][m] = ld_cluster_f32(rb_addr + 4u * (uint32_t)(m * kRows));
          }
#pragma unroll
        for (int u = 0; u < kR; ++u)
          if (r0 + u < p.cluster) {
#pragma unroll
            for (int m = 0; m < M; ++m) sum[m] += v[u][m];
          }
      }
      write_row<M>(p, n, sum, sc);
    }
    cluster_sync_all();
  } else if (complete) {
    write_row<M>(p, n, acc, sc);
  } else {
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
      // several contributors at a time: their loads are independent, the adds stay in
      // CTA order
      constexpr int kU = M <= 2 ? 8 : (M <= 8 ? 4 : 2);
      for (int64_t i = i_first; i <= i_last; i += kU) {
        float part[kU][M];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int64_t ci = i + u;
          if (ci <= i_last) {
            const int sl = (range_begin(ci, p.W, p.G) / T == rb) ? 0 : 1;
            const float* src = p.ws + (ci * 2 + sl) * (kRows * kMaxTokens);
#pragma unroll
            for (int m = 0; m < M; ++m) part[u][m] = __ldcg(src + m * kRows + tid);
          }
        }
#pragma unroll
        for (int u = 0; u < kU; ++u)
          if (i + u <= i_last) {
#pragma unroll
            for (int m = 0; m < M; ++m) sum[m] += part[u][m];
          }
      }
      write_row<M>(p, n, sum, sc);
      if (tid == 0) atomicExch(ctr, 0);
    }
    named_bar_sync(1, kConsumerWarps * 32);
  }
}

// Thread-per-row kernel (any M <= kMaxTokens): the four consumer warps share each chunk,
// thread r owning row r; its first value is found by a popc prefix sum over the chunk's
// masks (warp scan plus the other warps' kept counts).
template <int M, int ES, bool CL>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) linear_cc_kernel(const LinearParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)p.slots * p.slot_bytes);
  uint64_t* empty = full + p.slots;
  volatile int* s_flag = reinterpret_cast<volatile int*>(empty + p.slots);
  volatile int* tag = s_flag + 4;
  const int T = p.T;
  const int slots = p.slots;
  int64_t w0, w1;
  uint32_t crank;
  cta_range(p, CL, &w0, &w1, &crank);

  if (tid == 0) {
    for (int s = 0; s < slots; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
      tag[s] = -1;
    }
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    produce<M, false>(p, smem, full, empty, tag, w0, w1, lane);
    return;
  }

  // -------------------------------------------------------------- consumers
  pdl_wait();  // y, the workspace and x belong to the stream order
  float acc[M];
#pragma unroll
  for (int m = 0; m < M; ++m) acc[m] = 0.f;
  bool dead = false;  // a bounded wait expired: keep the barrier schedule, skip the math
  const int64_t rb_first = w0 / T;
  int64_t rb = rb_first;
  int t = (int)(w0 % T);
  int s = 0;
  uint32_t ph = 0;
  for (int64_t w = w0; w < w1; ++w) {
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
      const uint64_t mk = masks[tid];
      const uint32_t lo = (uint32_t)mk, hi = (uint32_t)(mk >> 32);
      const int plo = __popc(lo), pc = plo + __popc(hi);
      int incl = pc;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += u;
      }
      const int base = kept_before_quarter(masks, warp, lane);
      uint32_t XL[(M + 1) / 2], XH[(M + 1) / 2];
      load_x<M>(slot, p.chunk_region, lane, XL, XH);
      row_dot<M, ES>(lo, hi, plo, pc, base + incl - pc, slot + kMaskBytes, XL, XH, acc);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
    if (++s == slots) {
      s = 0;
      ph ^= 1u;
    }

    // ------------------------------------------------------------ row-block end
    const int t_cur = t;
    const int64_t rb_cur = rb;
    if (++t == T) {
      t = 0;
      ++rb;
    }
    if (t_cur != T - 1 && w + 1 != w1) continue;
    row_block_end<M, ES, CL>(p, smem, s_flag, acc, rb_cur, rb_cur * T >= w0 && t_cur == T - 1,
                             rb_cur == rb_first ? 0 : 1, crank, tid);
    // (a clustered CTA covers one row block: this was its last item)
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] = 0.f;
  }
}

// ---------------------------------------------------------------- asynchronous row-block end
// (warp-per-chunk kernel, stream-K): each warp flushes its partials into a double-buffered
// combine area and the last of the four to flush adds them and runs the epilogue alone
// while the others go on with the next row block.
struct FlushCtl {
  int flushed[2];  // warps that have flushed the row block held by buffer b
  int ready[2];    // local row block that may be written into buffer b next
};

// Rows 4*lane + i of row block rb: y = bf16(s * scale)
template <int M, int ES>
__device__ __forceinline__ void store_rows(const LinearParams& p, const float (&s)[4][M], int64_t rb, int lane) {
  // rows 4l .. 4l+3 of this lane: the pairs (4l, 4l+1) and (4l+2, 4l+3) of the pair product
  // are both in the lane
  const int64_t n0 = rb * kRows + 4 * lane;
  float sc[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) sc[i] = (ES == 1 && n0 + i < p.N) ? p.scale[n0 + i] : 1.f;
  if (p.epi == SP_EPI_PAIR_PRODUCT) {
    const int64_t ldy = p.N >> 1;
#pragma unroll
    for (int i = 0; i < 4; i += 2) {
      const int64_t n = n0 + i;
      if (n < p.N) {
#pragma unroll
        for (int m = 0; m < M; ++m) {
          const float g = bf16_bits_to_float(float_to_bf16_bits_rn(s[i][m] * sc[i]));
          const float u = bf16_bits_to_float(float_to_bf16_bits_rn(s[i + 1][m] * sc[i + 1]));
          p.y[(int64_t)m * ldy + (n >> 1)] = float_to_bf16_bits_rn(g * u);
        }
      }
    }
    return;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t n = n0 + i;
    if (n < p.N) {
      if (p.epi == SP_EPI_RESIDUAL) {
        const float rv = bf16_bits_to_float(p.r[n]);
#pragma unroll
        for (int m = 0; m < M; ++m) {
          uint16_t* yp = p.y + (int64_t)m * p.N + n;
          const float a = bf16_bits_to_float(float_to_bf16_bits_rn(s[i][m] * sc[i]));
          *yp = float_to_bf16_bits_rn((bf16_bits_to_float(__ldcg(reinterpret_cast<const unsigned short*>(yp))) + a) + rv);
        }
      } else {
#pragma unroll
        for (int m = 0; m < M; ++m) p.y[(int64_t)m * p.N + n] = float_to_bf16_bits_rn(s[i][m] * sc[i]);
      }
    }
  }
}

// End of row block rb run by one warp (rows 4*lane + i): a CTA that covered the whole row
// block writes y; otherwise it stores its partial in workspace slot `my_slot` and the last
// of the row block's CTAs to arrive adds the partials in CTA order and writes y.
template <int M, int ES>
__device__ __forceinline__ void row_block_end_warp(const LinearParams& p, const float (&sum)[4][M], int64_t rb,
                                                   bool complete, int my_slot, int lane) {
  if (complete) {
    store_rows<M, ES>(p, sum, rb, lane);
    return;
  }
  const int T = p.T;
  float* wsp = p.ws + ((int64_t)blockIdx.x * 2 + my_slot) * (kRows * kMaxTokens) + 4 * lane;
#pragma unroll
  for (int m = 0; m < M; ++m)
    __stcg(reinterpret_cast<float4*>(wsp + m * kRows), make_float4(sum[0][m], sum[1][m], sum[2][m], sum[3][m]));
  __threadfence();
  __syncwarp();
  const int64_t seg_begin = rb * T;
  const int64_t i_first = owner_of(seg_begin, p.W, p.G);
  const int64_t i_last = owner_of(seg_begin + T - 1, p.W, p.G);
  const int sf = (range_begin(i_first, p.W, p.G) / T == rb) ? 0 : 1;
  int* ctr = p.cnt + i_first * 2 + sf;
  int last = 0;
  if (lane == 0) last = (atomicAdd(ctr, 1) == (int)(i_last - i_first)) ? 1 : 0;
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) return;
  __threadfence();
  float tot[4][M];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int m = 0; m < M; ++m) tot[i][m] = 0.f;
  // several contributors at a time: their loads are independent, the adds stay in CTA order
  constexpr int kU = M <= 2 ? 4 : 1;
  for (int64_t i = i_first; i <= i_last; i += kU) {
    float4 part[kU][M];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t ci = i + u;
      if (ci <= i_last) {
        const int sl = (range_begin(ci, p.W, p.G) / T == rb) ? 0 : 1;
        const float* src = p.ws + (ci * 2 + sl) * (kRows * kMaxTokens) + 4 * lane;
#pragma unroll
        for (int m = 0; m < M; ++m) part[u][m] = __ldcg(reinterpret_cast<const float4*>(src + m * kRows));
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u)
      if (i + u <= i_last) {
#pragma unroll
        for (int m = 0; m < M; ++m) {
          tot[0][m] += part[u][m].x;
          tot[1][m] += part[u][m].y;
          tot[2][m] += part[u][m].z;
          tot[3][m] += part[u][m].w;
        }
      }
  }
  store_rows<M, ES>(p, tot, rb, lane);
  if (lane == 0) atomicExch(ctr, 0);
}

// Warp `warp` is done with local row block k of its CTA: its partial sums go to buffer
// k % 2, and the last of the kConsumerWarps warps to flush k adds them in warp order and
// runs the row block's end.
template <int M, int ES>
__device__ __forceinline__ void flush_async(const LinearParams& p, FlushCtl* ctl, float* comb,
                                            const float (&acc)[4][M], int k, int64_t rb_first, int64_t w0,
                                            int64_t w1, int warp, int lane) {
  const int T = p.T;
  const int b = k & 1;
  volatile int* ready = ctl->ready;
  if (ready[b] != k) {
    // the buffer still holds row block k - 2, whose end is under way
    const uint64_t t0 = global_ns();
    while (ready[b] != k) {
      __nanosleep(64);
      if (global_ns() - t0 > p.timeout_ns) {
        set_status(p.status, kStatusTimeout);
        break;
      }
    }
  }
  float* cb = comb + (size_t)b * kConsumerWarps * M * kRows;
#pragma unroll
  for (int m = 0; m < M; ++m)
    *reinterpret_cast<float4*>(cb + (warp * M + m) * kRows + 4 * lane) =
        make_float4(acc[0][m], acc[1][m], acc[2][m], acc[3][m]);
  __syncwarp();
  int last = 0;
  if (lane == 0) {
    __threadfence_block();
    last = (atomicAdd(&ctl->flushed[b], 1) == kConsumerWarps - 1) ? 1 : 0;
  }
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) return;
  __threadfence_block();
  float sum[4][M];
#pragma unroll
  for (int m = 0; m < M; ++m) {
    float4 a = *reinterpret_cast<const float4*>(cb + m * kRows + 4 * lane);
#pragma unroll
    for (int c = 1; c < kConsumerWarps; ++c) {
      const float4 v = *reinterpret_cast<const float4*>(cb + (c * M + m) * kRows + 4 * lane);
      a.x += v.x;
      a.y += v.y;
      a.z += v.z;
      a.w += v.w;
    }
    sum[0][m] = a.x;
    sum[1][m] = a.y;
    sum[2][m] = a.z;
    sum[3][m] = a.w;
  }
  __syncwarp();
  if (lane == 0) ctl->flushed[b] = 0;
  const int64_t rb = rb_first + k;
  row_block_end_warp<M, ES>(p, sum, rb, rb * T >= w0 && (rb + 1) * T <= w1, k == 0 ? 0 : 1, lane);
  __syncwarp();
  if (lane == 0) {
    __threadfence_block();
    ready[b] = k + 2;
  }
}

// Warp-per-chunk kernel (M <= 4): consumer warp c takes items c, c + 4, c + 8, ... of
// the CTA's range, and lane l owns rows 4l .. 4l+3 of its chunk, so one warp scan finds
// every row's first value and each ring slot is released by the one warp that read it;
// sixteen chunks per SM are in flight in the consumers instead of four.  At each row
// block's end the four warps' partial sums meet in shared memory and are added in warp
// order (deterministic): in stream-K mode by the last warp to get there, which runs the
// row block's end alone while the others go on (flush_async); in cluster mode, where a
// CTA's one row block ends with its range, by thread r <-> row r after a barrier.
template <int M, int ES, bool CL, bool PROBE = false, int OCC = kCtasPerSm>
__global__ void __launch_bounds__(kThreads, OCC) linear_ccw_kernel(const LinearParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)p.slots * p.slot_bytes);
  uint64_t* empty = full + p.slots;
  volatile int* s_flag = reinterpret_cast<volatile int*>(empty + p.slots);
  volatile int* tag = s_flag + 4;
  float* comb = reinterpret_cast<float*>(smem + p.comb_off);  // [2][kConsumerWarps][M][kRows]
  FlushCtl* fctl = reinterpret_cast<FlushCtl*>(comb + (CL ? 1 : 2) * kConsumerWarps * M * kRows);
  // PROBE (the failure-path test only): a barrier that nothing completes, in the unused upper
  // half of the 16-byte flag area (8-byte aligned: it follows the mbarrier arrays)
  uint64_t* probe = reinterpret_cast<uint64_t*>(const_cast<int*>(s_flag) + 2);
  const int T = p.T;
  const int slots = p.slots;  // >= kConsumerWarps
  int64_t w0, w1;
  uint32_t crank;
  cta_range(p, CL, &w0, &w1, &crank);

  if (tid == 0) {
    for (int s = 0; s < slots; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      tag[s] = -1;
    }
    for (int b = 0; b < 2; ++b) {
      fctl->flushed[b] = 0;
      fctl->ready[b] = b;
    }
    if constexpr (PROBE) mbar_init(probe, 1);
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    produce<M, OCC != kCtasPerSm>(p, smem, full, empty, tag, w0, w1, lane);
    return;
  }

  pdl_wait();
  if constexpr (OCC != kCtasPerSm) pdl_launch_dependents();
  bool dead = false;
  if (PROBE && blockIdx.x == 0 && warp == 0) {
    // failure-path test: a bounded wait on a barrier that nothing completes and no copy
    // targets; its expiry is recorded in the status word like any other, and the warp then
    // goes on normally (every copy it consumes has landed, so the results stay correct)
    if (!__all_sync(0xffffffffu, mbar_wait(probe, 0, p.probe_ns))) set_status(p.status, kStatusTimeout);
  }
  int s = warp;  // ring slot of this warp's next item (item n uses slot n % slots)
  uint32_t ph = 0;
  int64_t w = w0 + warp;
  const int64_t rb_first = w0 / T;
  const int64_t rb_last = w1 > w0 ? (w1 - 1) / T : rb_first - 1;
  for (int64_t rb = rb_first; rb <= rb_last; ++rb) {
    const int64_t wb = rb * T > w0 ? rb * T : w0;
    const int64_t we = (rb + 1) * T < w1 ? (rb + 1) * T : w1;
    float acc[4][M];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int m = 0; m < M; ++m) acc[i][m] = 0.f;
    for (; w < we; w += kConsumerWarps) {
      if (!dead && tag[s] != (int)(w - w0)) {
        // the slot may still hold an earlier item of another warp: wait until the producer
        // has claimed it for this one (it does so only once that item was consumed), so
        // the parity wait below cannot match an older phase of the slot's barrier
        const uint64_t t0 = global_ns();
        while (tag[s] != (int)(w - w0)) {
          __nanosleep(32);
          if (global_ns() - t0 > p.timeout_ns) {
            dead = true;
            set_status(p.status, kStatusTimeout);
            break;
          }
        }
        dead = __any_sync(0xffffffffu, dead);
      }
      if (!dead) {
        const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[s], ph, p.timeout_ns));
        if (!ok) {
          dead = true;
          set_status(p.status, kStatusTimeout);
        }
      }
      if (!dead) {
        const uint8_t* slot = smem + (size_t)s * p.slot_bytes;
        // masks of rows 4l .. 4l+3: two 16-byte loads
        const uint4 ma = *reinterpret_cast<const uint4*>(slot + 32 * lane);
        const uint4 mb = *reinterpret_cast<const uint4*>(slot + 32 * lane + 16);
        const uint32_t lo[4] = {ma.x, ma.z, mb.x, mb.z}, hi[4] = {ma.y, ma.w, mb.y, mb.w};
        int plo[4], pc[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          plo[i] = __popc(lo[i]);
          pc[i] = plo[i] + __popc(hi[i]);
        }
        const int tot = pc[0] + pc[1] + pc[2] + pc[3];
        int incl = tot;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
          const int u = __shfl_up_sync(0xffffffffu, incl, d);
          if (lane >= d) incl += u;
        }
        int e = incl - tot;  // first value of row 4l
        uint32_t XL[(M + 1) / 2], XH[(M + 1) / 2];
        load_x<M>(slot, p.chunk_region, lane, XL, XH);
        const uint8_t* vals = slot + kMaskBytes;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          row_dot<M, ES>(lo[i], hi[i], plo[i], pc[i], e, vals, XL, XH, acc[i]);
          e += pc[i];
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[s]);
      if ((s += kConsumerWarps) >= slots) {
        s -= slots;
        ph ^= 1u;
      }
    }
    if constexpr (!CL) {
      flush_async<M, ES>(p, fctl, comb, acc, (int)(rb - rb_first), rb_first, w0, w1, warp, lane);
    } else {
      // the four warps' partials for rows 4l + i, added in warp order by thread r <-> row r
#pragma unroll
      for (int m = 0; m < M; ++m)
        *reinterpret_cast<float4*>(comb + (warp * M + m) * kRows + 4 * lane) =
            make_float4(acc[0][m], acc[1][m], acc[2][m], acc[3][m]);
      named_bar_sync(2, kConsumerWarps * 32);
      float sum[M];
#pragma unroll
      for (int m = 0; m < M; ++m) {
        sum[m] = comb[m * kRows + tid];
#pragma unroll
        for (int c = 1; c < kConsumerWarps; ++c) sum[m] += comb[(c * M + m) * kRows + tid];
      }
      named_bar_sync(2, kConsumerWarps * 32);  // comb is rewritten at the next row block
      row_block_end<M, ES, CL>(p, smem, s_flag, sum, rb, wb == rb * T && we == (rb + 1) * T,
                               rb == rb_first ? 0 : 1, crank, tid);
    }
  }
}

// kind 0: thread-per-row kernel; kind 1: warp-per-chunk kernel (M <= 4)
template <int M, int ES>
sp_status launch_one(const LinearParams& p, cudaStream_t stream, size_t smem, int kind, int occ, bool pdl) {
  void (*kern)(const LinearParams);
  if constexpr (M <= 4) {
    if (occ == kCtasPerSmM1 || occ == kCtasPerSmM1b) {
      if constexpr (M == 1) {
        if (kind != 1 || p.cluster < 2 || p.probe_ns != 0) return SP_ERR_UNSUPPORTED;
        kern = occ == kCtasPerSmM1 ? linear_ccw_kernel<1, ES, true, false, kCtasPerSmM1>
                                   : linear_ccw_kernel<1, ES, true, false, kCtasPerSmM1b>;
      } else {
        return SP_ERR_UNSUPPORTED;
      }
    } else if (kind == 1 && p.probe_ns != 0) {
      if constexpr (ES == 2)
        kern = p.cluster > 1 ? linear_ccw_kernel<M, ES, true, true> : linear_ccw_kernel<M, ES, false, true>;
      else
        return SP_ERR_UNSUPPORTED;
    } else if (kind == 1)
      kern = p.cluster > 1 ? linear_ccw_kernel<M, ES, true> : linear_ccw_kernel<M, ES, false>;
    else
      kern = p.cluster > 1 ? linear_cc_kernel<M, ES, true> : linear_cc_kernel<M, ES, false>;
  } else {
    kern = p.cluster > 1 ? linear_cc_kernel<M, ES, true> : linear_cc_kernel<M, ES, false>;
  }
  static bool configured[5][2][kMaxDevices] = {};  // kernel attributes, once per device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= kMaxDevices) return SP_ERR_UNSUPPORTED;
  const int ci = p.cluster > 1 ? 1 : 0;
  // the probe variant and the six- and five-CTA variants are kernels of their own
  const int ki = occ == kCtasPerSmM1 ? 3 : occ == kCtasPerSmM1b ? 4 : p.probe_ns != 0 ? 2 : kind;
  if (!configured[ki][ci][dev]) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemOptIn) != cudaSuccess ||
        (ci && cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)) {
      cudaGetLastError();
      return SP_ERR_CUDA;
    }
    configured[ki][ci][dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.G);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  int na = 1;
  if (p.cluster > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)p.cluster;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    na = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  if (cudaLaunchKernelEx(&cfg, kern, p) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  return SP_OK;
}

template <int ES>
sp_status dispatch_m(const LinearParams& p, cudaStream_t stream, size_t smem, int kind, int occ, bool pdl) {
  switch (p.M) {
    case 1: return launch_one<1, ES>(p, stream, smem, kind, occ, pdl);
    case 2: return launch_one<2, ES>(p, stream, smem, kind, occ, pdl);
    case 3: return launch_one<3, ES>(p, stream, smem, kind, occ, pdl);
    case 4: return launch_one<4, ES>(p, stream, smem, kind, occ, pdl);
    case 5: return launch_one<5, ES>(p, stream, smem, kind, occ, pdl);
    case 6: return launch_one<6, ES>(p, stream, smem, kind, occ, pdl);
    case 7: return launch_one<7, ES>(p, stream, smem, kind, occ, pdl);
    case 8: return launch_one<8, ES>(p, stream, smem, kind, occ, pdl);
    case 9: return launch_one<9, ES>(p, stream, smem, kind, occ, pdl);
    case 10: return launch_one<10, ES>(p, stream, smem, kind, occ, pdl);
    case 11: return launch_one<11, ES>(p, stream, smem, kind, occ, pdl);
    case 12: return launch_one<12, ES>(p, stream, smem, kind, occ, pdl);
    case 13: return launch_one<13, ES>(p, stream, smem, kind, occ, pdl);
    case 14: return launch_one<14, ES>(p, stream, smem, kind, occ, pdl);
    case 15: return launch_one<15, ES>(p, stream, smem, kind, occ, pdl);
    case 16: return launch_one<16, ES>(p, stream, smem, kind, occ, pdl);
    default: return SP_ERR_INVALID_ARG;
  }
}

// Thread-block cluster split: each row block is split over S CTAs of one cluster, which
// replaces the global split-K fix-up by a distributed-shared-memory reduction; S = 1 is the
// stream-K launch over grid_cc CTAs, taken only when not even two CTAs per row block fit
// the SMs' CTA slots.  S is the largest cluster size that fits the slots (occ CTAs per
// SM) and leaves each CTA at least cmin chunks (at least two ranks when the row block is
// short), from 2..8 and 16.  Measured on GB300 (decode steps of the 32-layer Llama-2-7B
// stack, 70%, bf16 and INT8): a step ran fastest when every launch's grid filled most of
// the slots, because each launch then overlaps evenly with its neighbours under
// programmatic dependent launch; small grids that won alone (q/k/v in 288 CTAs instead
// of 576) cost up to 6 us per layer in the step.  With four CTAs per SM, 4-chunk CTAs (o,
// S = 16) lost to 8-chunk ones (cmin = 8); with six they won (cmin = 4).  Cluster sizes
// 9..15 ran 35% slower than 8 on down and are not taken.  Choices: four CTAs per SM --
// q/k/v (96 row blocks) 6, o (32) 8, gate/up (172) 3, down (32 of 172 chunks) 16; six --
// 8, 16, 5, 16.
int cluster_cc(const sp_matrix* h, int occ) {
  const int64_t rb = std::max<int32_t>(h->RB, 1);
  const int64_t T = h->T;
  const int64_t smax = std::min<int64_t>(std::min<int64_t>(16, (int64_t)occ * h->num_sms / rb), T);
  if (smax < 2) return 1;
  const int64_t cmin = std::min<int64_t>(occ == kCtasPerSm ? 8 : 4, (T + 1) / 2);
  for (int64_t S = smax; S > 2; --S) {
    if (S > 8 && S < 16) continue;
    if ((T + S - 1) / S >= cmin) return (int)S;
  }
  return 2;
}

int grid_cc(const sp_matrix* h) {
  const int64_t W = (int64_t)h->RB * h->T;
  static_assert(kCtasPerSm <= kMaxGridPerSm, "grid must fit the workspace counter region");
  // at least ~6 chunks per CTA, whole multiples of the SM count while W allows
  const int64_t per_sm = std::max<int64_t>(1, std::min<int64_t>(kCtasPerSm, W / ((int64_t)h->num_sms * 6)));
  return (int)std::min<int64_t>(per_sm * h->num_sms, W);
}

// Shared-memory plan of one launch with Mt batch rows: ring slots, whether the
// warp-per-chunk kernel runs (M <= 4 and room for a slot per consumer warp after its
// partials), and the offsets of the warps' partials and of the cluster partial.
struct CcPlan {
  int slots, kind, occ;
  uint32_t slot_bytes, comb_off, part_off;
  size_t smem;
};
bool cc_plan(const sp_matrix* h, int Mt, int S, int occ, CcPlan* pl) {
  const uint32_t chunk_region = (uint32_t)((h->max_chunk + 127) / 128 * 128);
  pl->slot_bytes = chunk_region + (uint32_t)Mt * 128u;
  // shared memory: ring slots, 2*slots mbarriers (<= 256 B), the flag (16 B), the slot
  // tags (<= 64 B), the warps' partials (warp-per-chunk kernel) and the CTA's FP32
  // partial (cluster mode)
  const size_t part_bytes = S > 1 ? (size_t)kRows * Mt * sizeof(float) : 0;
  // stream-K double-buffers the warps' partials (a warp may reach the next row block's end
  // while the last one's is still being summed); a cluster CTA ends one row block
  const size_t comb_bytes = (S > 1 ? 1 : 2) * (size_t)kConsumerWarps * kRows * Mt * sizeof(float) + sizeof(FlushCtl);
  pl->kind = 0;
  pl->occ = occ;
  size_t ring = (occ == kCtasPerSmM1 ? kSmemBudgetM1 : occ == kCtasPerSmM1b ? kSmemBudgetM1b : kSmemBudget) - 256 -
                16 - 64 - part_bytes;
  if (Mt <= 4 && (ring - comb_bytes) / pl->slot_bytes >= (size_t)kConsumerWarps) {
    pl->kind = 1;
    ring -= comb_bytes;
  }
  pl->slots = (int)std::min<size_t>(16, ring / pl->slot_bytes);
  if (pl->slots < 2 || (occ != kCtasPerSm && pl->kind != 1)) return false;
  pl->comb_off = (uint32_t)(((size_t)pl->slots * pl->slot_bytes + 2 * (size_t)pl->slots * 8 + 16 +
                             4 * (size_t)pl->slots + 15) /
                            16 * 16);
  pl->part_off = pl->comb_off + (uint32_t)(pl->kind == 1 ? comb_bytes : 0);
  pl->smem = pl->part_off + part_bytes;
  return true;
}

// The launch configuration of one launch with Mt batch rows: six CTAs per SM for a
// warp-per-chunk cluster launch at M = 1 where its plan fits, else five where that fits,
// else four; S = 1 (stream-K) without clusters.
bool select_cc(const sp_matrix* h, int Mt, bool allow_cluster, bool probe, int* S, CcPlan* pl) {
  if (allow_cluster && Mt == 1 && !probe) {
    for (const int occ : {kCtasPerSmM1, kCtasPerSmM1b}) {
      const int s1 = cluster_cc(h, occ);
      if (s1 > 1 && cc_plan(h, 1, s1, occ, pl)) {
        *S = s1;
        return true;
      }
    }
  }
  *S = allow_cluster ? cluster_cc(h, kCtasPerSm) : 1;
  return cc_plan(h, Mt, *S, kCtasPerSm, pl);
}

}  // namespace

int cc_kernel_kind(const sp_matrix* h, int64_t M) {
  CcPlan pl;
  int S;
  return select_cc(h, (int)std::min<int64_t>(kMaxTokens, M), true, false, &S, &pl) ? pl.kind : -1;
}

size_t workspace_bytes_cc(const sp_matrix* h, int64_t /*M*/) {
  const size_t G = (size_t)grid_cc(h);
  return ws_counter_bytes(h->num_sms) + 2 * G * kRows * kMaxTokens * sizeof(float);
}

sp_status launch_linear_cc(const sp_matrix* h, const uint16_t* x, int64_t M, uint16_t* y, void* ws, size_t ws_bytes,
                           cudaStream_t stream, bool allow_cluster, uint64_t probe_ns, int32_t epi,
                           const uint16_t* r) {
  // the configuration depends on the batch rows of a launch: full launches of kMaxTokens
  // rows and one ragged tail; the workspace is checked before the first launch
  const bool probe = probe_ns != 0;
  auto stream_k = [&](int Mt) {
    CcPlan q;
    int S = 1;
    return !select_cc(h, Mt, allow_cluster, probe, &S, &q) || S == 1;
  };
  const int tail = (int)(M % kMaxTokens);
  const bool needs_ws = (M >= kMaxTokens && stream_k(kMaxTokens)) || (tail != 0 && stream_k(tail));
  const size_t need = workspace_bytes_cc(h, M);
  if (needs_ws && (!ws || ws_bytes < need)) return SP_ERR_WORKSPACE;
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
  p.cnt = reinterpret_cast<int*>(ws);
  p.ws = ws ? reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(ws) + ws_counter_bytes(h->num_sms)) : nullptr;
  p.timeout_ns = wait_timeout_ns();
  p.probe_ns = probe_ns;
  p.epi = epi;
  p.r = r;
  const int64_t ldy = epi == SP_EPI_PAIR_PRODUCT ? h->N / 2 : h->N;
  p.chunk_region = (uint32_t)((h->max_chunk + 127) / 128 * 128);
  for (int64_t m0 = 0; m0 < M; m0 += kMaxTokens) {
    const int Mt = (int)std::min<int64_t>(kMaxTokens, M - m0);
    int S = 1;
    CcPlan pl;
    if (!select_cc(h, Mt, allow_cluster, probe, &S, &pl)) return SP_ERR_UNSUPPORTED;
    p.M = Mt;
    p.cluster = S;
    p.G = S > 1 ? h->RB * S : grid_cc(h);
    p.x = x + m0 * h->K;
    p.y = y + m0 * ldy;
    p.slot_bytes = pl.slot_bytes;
    p.slots = pl.slots;
    p.comb_off = pl.comb_off;
    p.part_off = pl.part_off;
    const int kind = pl.kind;
    const size_t smem = pl.smem;
    // after an in-place weight update the first launch waits for the whole previous grid
    // (no weight copy may start before its writes are visible)
    const bool pdl = !(m0 == 0 && h->weights_written);
    const sp_status st = h->esize == 2 ? dispatch_m<2>(p, stream, smem, kind, pl.occ, pdl)
                                        : dispatch_m<1>(p, stream, smem, kind, pl.occ, pdl);
    if (st != SP_OK) return st;
    h->weights_written = 0;
  }
  return SP_OK;
}

}  // namespace sp
