// sp_linear_tc.cu -- sparse linear on the 5th-generation tensor cores (tcgen05).
//
// The GPU engine of Sec. 2.4.2: compressed submatrices move from global memory onto
// the chip, are expanded by their bitmask, and the tensor cores run on the expanded
// tiles at the dense rate while global traffic stays at the compressed size.  On
// sm_103a the expanded tile goes to tensor memory and feeds tcgen05.mma directly:
//
//   D[128 rows, Ntok tokens] (fp32, TMEM) += A[128 rows, 64 k] (bf16, TMEM) x B[64 k, Ntok]
//
// where A is one chunk (128 weight rows x one 64-wide K-tile) expanded by its masks and
// B is x[tokens, 64t : 64t+64) brought in by TMA (128-byte swizzle, K-major).
//
// CTA (one per SM, persistent, stream-K over work items (token tile, row block, K-tile)):
//   warp 0 lane 0   producer: cp.async.bulk of each chunk and a TMA tile of x into a
//                   ring of S shared-memory slots; item n uses slot n % S and TMEM A
//                   stage n % S, and one MMA commit frees both (stage_free[n % S]);
//   warp 1          TMEM allocation; lane 0 issues the MMAs (4 x K=16 per chunk) and
//                   commits them to mbarriers that free the stage and, at a segment's
//                   end, hand D to the epilogue;
//   warps 2-..      EG expander warpgroups taking chunks round-robin: thread r of a
//                   warpgroup owns TMEM lane / chunk row r; it finds its first value by a
//                   popc prefix sum, expands 64 columns into 32 bf16x2 registers, and
//                   stores them to an A stage with tcgen05.st; at a row-block end the
//                   warpgroup that expanded the last K-tile reads D with tcgen05.ld and
//                   writes bf16 y (RNE), or an FP32 partial for the deterministic
//                   stream-K fix-up shared with the CUDA-core kernel.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "sp_internal.cuh"

namespace sp {
namespace {

// Expander warpgroups EG (a template parameter: 2 or 3) take items round-robin; a CTA
// runs 2 + 4 * EG warps.  Three groups (14 warps: three expander warps on each SM
// sub-partition, at most 128 registers) for token tiles of up to 64 tokens, where the
// ring still holds two slots per group: at M = 16 the kernel with two groups issued on
// 42 % of cycles, stalled on fixed-latency and shared-memory results with 10 warps per
// SM (ncu).  Two groups for wider tiles (their x tiles leave room for few slots).  Four
// groups (18 warps) would put five warps on two sub-partitions, whose 16K registers then
// allow 96 per thread: ~300 bytes of spills.
constexpr int kMaxExpGroups = 3;
__host__ __device__ constexpr int tc_threads(int eg) { return (2 + 4 * eg) * 32; }
constexpr int kExpWarp0 = 2;          // first expander warp
constexpr int kMaxAStages = 16;       // A tiles in TMEM (32 columns each), at most
constexpr int kMaxDBufs = 2;          // D accumulators in TMEM (ntok columns each), at most
constexpr int kMaxNtok = 256;         // tokens per tile (MMA N)
constexpr uint32_t kTmemCols = 512;   // nD x D (ntok rounded to 32 columns) + nA x 32 A columns
constexpr size_t kSmemLimit = 226 * 1024;
constexpr int kMaxDevices = 64;
constexpr int kMaxSlots = 16;

// ------------------------------------------------------------------ tcgen05 / TMA wrappers
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_store32(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]),
      "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]),
      "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
}
__device__ __forceinline__ void tmem_store_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_load32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
        "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_load_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// D[tmem] (+)= A[tmem] * B[smem desc]; bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_ts(uint32_t d_taddr, uint32_t a_taddr, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_taddr),
      "r"(a_taddr), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
// TMA tile store shared -> global (bulk group); rows/columns past the tensor are clipped.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1)
               : "memory");
}
// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row atoms of
// 1024 bytes stacked along M/N (stride byte offset 1024), atom base 1024-byte aligned.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);        // start address
  d |= (uint64_t)1u << 16;                        // leading byte offset (unused for SW128 K-major)
  d |= (uint64_t)((1024u >> 4) & 0x3FFFu) << 32;  // stride byte offset
  d |= (uint64_t)1u << 46;                        // descriptor version (sm_100 family)
  d |= (uint64_t)2u << 61;                        // swizzle mode: 128B
  return d;
}
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major, M = 128.
__host__ __device__ constexpr uint32_t idesc_bf16(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

__device__ __forceinline__ uint16_t i8_to_bf16(uint32_t byte) {
  const float f = __uint_as_float(0x4B000000u | (byte ^ 0x80u)) - 8388736.0f;
  return (uint16_t)(__float_as_uint(f) >> 16);
}

// One output word (two adjacent columns) of a row's expansion, bf16 values: each kept
// column takes the next value of the stream at shared address `pa` (which advances);
// a dropped column gives +0.  Written in PTX so every column is one predicate-setting
// AND, one predicated 16-bit shared load and one predicated pointer increment.
template <uint32_t B0, uint32_t B1>
__device__ __forceinline__ uint32_t expand_word_bf16(uint32_t m, uint32_t& pa) {
  uint32_t o;
  asm("{\n\t.reg .pred p0, p1;\n\t.reg .b32 t0, t1, lo, hi;\n\t"
      "and.b32 t0, %2, %3;\n\t"
      "setp.ne.b32 p0, t0, 0;\n\t"
      "and.b32 t1, %2, %4;\n\t"
      "setp.ne.b32 p1, t1, 0;\n\t"
      "mov.b32 lo, 0;\n\t"
      "mov.b32 hi, 0;\n\t"
      "@p0 ld.shared.u16 lo, [%1];\n\t"
      "@p0 add.u32 %1, %1, 2;\n\t"
      "@p1 ld.shared.u16 hi, [%1];\n\t"
      "@p1 add.u32 %1, %1, 2;\n\t"
      "prmt.b32 %0, lo, hi, 0x5410;\n\t}"
      : "=r"(o), "+r"(pa)
      : "r"(m), "n"(B0), "n"(B1));
  return o;
}
// The same for int8 values (one byte each), converted exactly to bf16.
template <uint32_t B0, uint32_t B1>
__device__ __forceinline__ uint32_t expand_word_i8(uint32_t m, uint32_t& pa) {
  uint32_t lo = 0, hi = 0;
  uint32_t b0, b1;
  asm("{\n\t.reg .pred p0, p1;\n\t.reg .b32 t0, t1;\n\t"
      "and.b32 t0, %3, %4;\n\t"
      "setp.ne.b32 p0, t0, 0;\n\t"
      "and.b32 t1, %3, %5;\n\t"
      "setp.ne.b32 p1, t1, 0;\n\t"
      "mov.b32 %0, 128;\n\t"
      "mov.b32 %1, 128;\n\t"
      "@p0 ld.shared.u8 %0, [%2];\n\t"
      "@p0 add.u32 %2, %2, 1;\n\t"
      "@p1 ld.shared.u8 %1, [%2];\n\t"
      "@p1 add.u32 %2, %2, 1;\n\t}"
      : "=r"(b0), "=r"(b1), "+r"(pa)
      : "r"(m), "n"(B0), "n"(B1));
  // a dropped column loads the byte 0x80 = -128 ... replaced below by +0
  lo = (m & B0) ? i8_to_bf16(b0) : 0u;
  hi = (m & B1) ? i8_to_bf16(b1) : 0u;
  return lo | (hi << 16);
}

template <int ES, int I>
__device__ __forceinline__ void expand_pair(uint32_t mlo, uint32_t mhi, uint32_t& pa, uint32_t& pb,
                                            uint32_t (&o)[32]) {
  constexpr uint32_t B0 = 1u << (2 * I), B1 = 1u << (2 * I + 1);
  if constexpr (ES == 2) {
    o[I] = expand_word_bf16<B0, B1>(mlo, pa);
    o[16 + I] = expand_word_bf16<B0, B1>(mhi, pb);
  } else {
    o[I] = expand_word_i8<B0, B1>(mlo, pa);
    o[16 + I] = expand_word_i8<B0, B1>(mhi, pb);
  }
  if constexpr (I + 1 < 16) expand_pair<ES, I + 1>(mlo, mhi, pa, pb, o);
}

struct TcParams {
  LinearParams p;     // shared fields (buf, off, scale, y, ws, cnt, status, N, K, T, RB, M, W, G, slots, ...)
  int32_t ntok;       // tokens per tile (MMA N), multiple of 16, <= 256
  int32_t mt;         // token tiles
  uint32_t b_bytes;   // bytes of one x tile in shared memory (ntok * 128)
  uint32_t chunk_off; // offset of the chunk region inside a slot
  int32_t n_a;        // A stages in TMEM (2..kMaxAStages)
  int32_t n_d;        // D buffers in TMEM (1..kMaxDBufs); segment k accumulates in buffer k % n_d
  uint32_t d_cols;    // TMEM columns per D buffer (ntok rounded up to 32)
  uint32_t a_col0;    // first TMEM column of the A stages (n_d * d_cols)
  int32_t y_tma;      // 1: y is written by TMA stores from a staging tile (needs N % 8 == 0)
  uint32_t stg_off;   // shared-memory offset of the staging tiles [EG][2][32][128] bf16
};

constexpr int kStgTokens = 32;                          // tokens per staged block
constexpr int kStgBox = 16;                             // tokens per TMA store box
constexpr uint32_t kStgBytes = kStgTokens * kRows * 2;  // one staging buffer

// Rows rb*128 + r (thread r of the warpgroup) for tokens tok0 .. tok0+nv-1 (nv <= 32, a
// multiple of 16) of y: bf16(val[i] * sc).  With a y tensor map the warpgroup writes the
// block into one of its two staging buffers and thread 0 stores it with TMA (16-token
// boxes; the hardware clips rows past M and columns past N); strided scalar stores of
// 2-byte values cost ~1.8 us per 32-token block.  Otherwise each thread stores its row.
__device__ __forceinline__ void store_y_block(const TcParams& tp, const CUtensorMap* tmap_y, uint16_t* stg, int& step,
                                              const float (&val)[32], float sc, int nv, int64_t tok0, int64_t rb,
                                              int r, int tid128, int bar) {
  const LinearParams& p = tp.p;
  if (tp.y_tma) {
    uint16_t* buf = stg + (size_t)(step & 1) * (kStgBytes / 2);
    if (tid128 == 0) bulk_wait_read<1>();  // the store that last read this buffer is done
    named_bar_sync(bar, 128);
#pragma unroll
    for (int i = 0; i < kStgTokens; ++i) buf[i * kRows + r] = float_to_bf16_bits_rn(val[i] * sc);
    fence_proxy_async_smem();
    named_bar_sync(bar, 128);
    if (tid128 == 0) {
      for (int b0 = 0; b0 < nv; b0 += kStgBox) tma_store_2d(tmap_y, buf + b0 * kRows, (int)(rb * kRows), (int)(tok0 + b0));
      bulk_commit();
    }
    ++step;
  } else {
    const int64_t nrow = rb * kRows + r;
#pragma unroll
    for (int i = 0; i < kStgTokens; ++i) {
      const int64_t tok = tok0 + i;
      if (i < nv && tok < p.M && nrow < p.N) p.y[tok * p.N + nrow] = float_to_bf16_bits_rn(val[i] * sc);
    }
  }
}

// TMEM split for a token tile of ntok columns: D buffers first, A stages after.  Small
// tiles (decode) leave room for two D buffers and up to 14 A stages, so neither the
// epilogue of one (row block, token tile) segment nor the tcgen05.commit round trip that
// frees an A stage stalls the MMA issuer.
__host__ __device__ inline void tmem_split(int ntok, int* n_a, int* n_d, uint32_t* d_cols) {
  const uint32_t dc = ((uint32_t)ntok + 31u) / 32u * 32u;
  const int nd = (2u * dc <= kTmemCols / 2) ? 2 : 1;
  int na = (int)((kTmemCols - (uint32_t)nd * dc) / 32u);
  if (na > kMaxAStages) na = kMaxAStages;
  *n_a = na;
  *n_d = nd;
  *d_cols = dc;
}

template <int ES, int EG>
__global__ void __launch_bounds__(tc_threads(EG), 1)
    linear_tc_kernel(const __grid_constant__ TcParams tp, const __grid_constant__ CUtensorMap tmap_x,
                     const __grid_constant__ CUtensorMap tmap_y) {
  extern __shared__ uint8_t smem_raw[];
  const LinearParams& p = tp.p;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int slots = p.slots;
  // Ring: item n uses slot n % S and A stage n % S (S = slots <= A stages, a multiple of EG).
  //   full[s]       chunk and x tile landed (producer's expect_tx + the copies)
  //   a_full[s]     the four warps of the item's expander warpgroup stored the A stage
  //   stage_free[s] the item's MMAs completed (one commit): slot and A stage are free.
  // The expanders read the chunk before arriving on a_full, and the MMAs are issued only
  // after a_full, so that one commit also covers the expanders' reads of the slot.  An
  // expander waits only on full[s]: the producer refills a slot only after stage_free,
  // and with S a multiple of EG a slot's previous item belongs to the same warpgroup.
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)slots * p.slot_bytes);
  uint64_t* stage_free = full + slots;
  uint64_t* a_full = stage_free + slots;
  // D handshakes.  Segment k (the k-th (token tile, row block) this CTA touches)
  // accumulates in buffer k % n_d, and its epilogue is run by the warpgroup that expanded
  // its last K-tile.  d_full has one barrier per (buffer, warpgroup): a group waits on
  // its own barriers one segment at a time, in order, so a parity wait can never match
  // an older phase (a group may reach the end of a short segment before the MMA issuer
  // has finished the previous segment on that buffer).  d_empty has one barrier per
  // buffer: the MMA issuer starts segment k only after the epilogue of segment k - n_d
  // has read that buffer, so those epilogues complete in order.
  uint64_t* d_full = a_full + slots;                      // [kMaxDBufs][EG]
  uint64_t* d_empty = d_full + kMaxDBufs * kMaxExpGroups; // [kMaxDBufs]
  uint32_t* tmem_base_slot = reinterpret_cast<uint32_t*>(d_empty + kMaxDBufs);
  volatile int* s_flag = reinterpret_cast<volatile int*>(tmem_base_slot + 1);  // one per warpgroup

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t w0 = range_begin(blockIdx.x, p.W, p.G);
  const int64_t w1 = range_begin(blockIdx.x + 1, p.W, p.G);
  const int T = p.T;
  const int64_t C = (int64_t)p.RB * T;  // chunks per token tile

  if (tid == 0) {
    for (int s = 0; s < slots; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&stage_free[s], 1);  // one MMA commit
      mbar_init(&a_full[s], 4);      // the four warps of an expander warpgroup
    }
    for (int b = 0; b < kMaxDBufs * EG; ++b) mbar_init(&d_full[b], 1);
    for (int b = 0; b < kMaxDBufs; ++b) mbar_init(&d_empty[b], 4);  // the epilogue warpgroup's four warps
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_base_slot, kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmap_x);
    if (tp.y_tma) prefetch_tmap(&tmap_y);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_base_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // The whole warp walks the items (it shares the offset window); lane 0 issues.
    const uint64_t pol = policy_evict_first();
    OffsetWindow ow;
    // item w = mtile * C + c, c = rb * T + t: walked with counters (no 64-bit division
    // on the issuing thread's critical path)
    int64_t c = w0 % C, mtile = w0 / C;
    int t = (int)(c % T);
    ow.init(p.off, C + 1, c);
    const int64_t n_pre = imin64((int64_t)slots, w1 - w0);
    for (int64_t i = 0, ci = c; i < n_pre; ++i) {  // weight bytes do not depend on the previous grid
      uint64_t o0, o1;
      ow.at(ci, &o0, &o1);
      if (++ci == C) ci = 0;
      if (lane == 0) {
        const uint32_t bytes = (uint32_t)(o1 - o0);
        mbar_arrive_expect_tx(&full[i], bytes + tp.b_bytes);
        bulk_g2s_hint(smem + (size_t)i * p.slot_bytes + tp.chunk_off, p.buf + o0, bytes, &full[i], pol);
      }
    }
    pdl_wait();
    pdl_launch_dependents();
    int s = 0;
    uint32_t ph = 0;
    bool failed = false;
    for (int64_t w = w0, n = 0; w < w1; ++w, ++n) {
      uint8_t* slot = smem + (size_t)s * p.slot_bytes;
      if (n >= n_pre) {
        uint64_t o0, o1;
        ow.at(c, &o0, &o1);
        if (lane == 0) {
          if (!mbar_wait(&stage_free[s], ph ^ 1u, p.timeout_ns)) {
            set_status(p.status, kStatusTimeout);
            failed = true;
          } else {
            const uint32_t bytes = (uint32_t)(o1 - o0);
            mbar_arrive_expect_tx(&full[s], bytes + tp.b_bytes);
            bulk_g2s_hint(slot + tp.chunk_off, p.buf + o0, bytes, &full[s], pol);
          }
        }
        failed = __shfl_sync(0xffffffffu, failed, 0);
        if (failed) break;
      }
      if (lane == 0) tma_load_2d(slot, &tmap_x, kTileK * t, (int)(mtile * tp.ntok), &full[s]);
      if (++s == slots) {
        s = 0;
        ph ^= 1u;
      }
      if (++t == T) t = 0;
      if (++c == C) {
        c = 0;
        ++mtile;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      pdl_wait();
      pdl_launch_dependents();
      const uint32_t idesc = idesc_bf16(tp.ntok);
      const int n_d = tp.n_d;
      int s = 0;
      uint32_t ph = 0;
      int k = -1;  // local segment number
      int db = 0;  // D buffer of segment k
      uint32_t d_taddr = tmem;
      bool dead = false;
      int t = (int)(w0 % T);  // K-tile of item w
      for (int64_t w = w0; w < w1; ++w) {
        const bool seg_first = (w == w0) || t == 0;
        const bool seg_last = (w + 1 == w1) || t == T - 1;
        if (++t == T) t = 0;
        if (seg_first) {
          ++k;
          db = k % n_d;
          d_taddr = tmem + (uint32_t)db * tp.d_cols;
          // D buffer reuse: wait for the (k / n_d - 1)-th completion of d_empty[db], the
          // epilogue of segment k - n_d
          if (!dead && k >= n_d) {
            if (!mbar_wait(&d_empty[db], (uint32_t)((k / n_d - 1) & 1), p.timeout_ns)) {
              dead = true;
              set_status(p.status, kStatusTimeout);
            }
          }
        }
        if (!dead && !mbar_wait(&full[s], ph, p.timeout_ns)) {
          dead = true;
          set_status(p.status, kStatusTimeout);
        }
        if (!dead && !mbar_wait(&a_full[s], ph, p.timeout_ns)) {
          dead = true;
          set_status(p.status, kStatusTimeout);
        }
        if (!dead) {
          tc_fence_after();
          const uint32_t b_saddr = smem_u32(smem + (size_t)s * p.slot_bytes);
          const uint32_t a_taddr = tmem + tp.a_col0 + (uint32_t)s * 32u;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t bdesc = smem_desc_sw128(b_saddr + (uint32_t)kk * 32u);
            mma_ts(d_taddr, a_taddr + (uint32_t)kk * 8u, bdesc, idesc, (seg_first && kk == 0) ? 0u : 1u);
          }
          mma_commit(&stage_free[s]);
          if (seg_last) mma_commit(&d_full[db * EG + (int)((w - w0) % EG)]);
        }
        if (++s == slots) {
          s = 0;
          ph ^= 1u;
        }
      }
    }
  } else {
    // ------------------------------------------------------------ expanders + epilogue
    pdl_wait();
    pdl_launch_dependents();
    const int grp = (warp - kExpWarp0) >> 2;  // this warpgroup takes items n = grp (mod 2)
    const int q = warp & 3;                   // TMEM lane quarter this warp may access
    const int r = q * 32 + lane;              // chunk row == TMEM lane
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const int tid128 = (warp - kExpWarp0 - 4 * grp) * 32 + lane;
    bool dead = false;
    const int64_t sg_first = w0 / T;
    // ring position of item n = grp, grp + EG, ... (slots a multiple of EG)
    int s = grp;
    uint32_t ph = 0;
    int t = (int)((w0 + grp) % T);  // K-tile of item w
    uint32_t dph_bits = 0;          // phase parity of this group's d_full barrier, per buffer
    uint16_t* stg = reinterpret_cast<uint16_t*>(smem + tp.stg_off) + (size_t)grp * kStgBytes;  // 2 buffers
    int stg_step = 0;
    const int bar = 1 + grp;        // named barrier of this warpgroup
    for (int64_t w = w0 + grp, n = grp; w < w1; w += EG, n += EG) {
      const bool seg_last = (w + 1 == w1) || t == T - 1;
      for (t += EG; t >= T;) t -= T;
      if (!dead) {
        const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[s], ph, p.timeout_ns));
        if (!ok) {
          dead = true;
          set_status(p.status, kStatusTimeout);
        }
      }
      if (!dead) {
        tc_fence_after();
        const uint8_t* chunk = smem + (size_t)s * p.slot_bytes + tp.chunk_off;
        const uint64_t* masks = reinterpret_cast<const uint64_t*>(chunk);
        const uint64_t mk = masks[r];
        const uint32_t mlo = (uint32_t)mk, mhi = (uint32_t)(mk >> 32);
        const int plo = __popc(mlo);
        const int pc = plo + __popc(mhi);
        int incl = pc;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
          const int u = __shfl_up_sync(0xffffffffu, incl, d);
          if (lane >= d) incl += u;
        }
        const int base = kept_before_quarter(masks, q, lane);
        const int e0 = base + incl - pc;
        // Static walk over the 64 columns: a kept column takes the next value of its
        // half's stream.  Columns 0-31 and 32-63 read two independent streams (the
        // second starts after the first half's plo values) for instruction-level
        // parallelism; each step is one predicate-setting AND, a predicated load and a
        // predicated pointer increment.
        uint32_t o[32];
        const uint32_t vbase = smem_u32(chunk + kMaskBytes);
        uint32_t pa = vbase + (uint32_t)(e0 * ES);   // stream of columns 0-31
        uint32_t pb = pa + (uint32_t)(plo * ES);     // stream of columns 32-63
        expand_pair<ES, 0>(mlo, mhi, pa, pb, o);
        tmem_store32(tmem + lane_base + tp.a_col0 + (uint32_t)s * 32u, o);
        tmem_store_wait();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[s]);
      if ((s += EG) >= slots) {
        s -= slots;
        ph ^= 1u;
      }

      // ---------------------------------------------------------- segment end: epilogue
      // Taken by the warpgroup that expanded the segment's last K-tile.
      if (!seg_last) continue;
      const int64_t sg = w / T;  // segment = (token tile, row block)
      const int64_t seg_begin = sg * T;
      const int64_t mtile = sg / p.RB;
      const int64_t rb = sg % p.RB;
      const int64_t nrow = rb * kRows + r;
      const float sc = (ES == 1 && nrow < p.N) ? p.scale[nrow] : 1.f;
      const int kseg = (int)(sg - sg_first);  // local segment number
      const int db = kseg % tp.n_d;
      const uint32_t dph = (dph_bits >> db) & 1u;
      dph_bits ^= 1u << db;
      const uint32_t d_taddr = tmem + (uint32_t)db * tp.d_cols;
      if (!dead) {
        const bool ok = __all_sync(0xffffffffu, mbar_wait(&d_full[db * EG + grp], dph, p.timeout_ns));
        if (!ok) {
          dead = true;
          set_status(p.status, kStatusTimeout);
        }
      }
      tc_fence_after();
      // this CTA ran the whole segment: its first and its last K-tile
      const bool complete = seg_begin >= w0 && (w + 1) % T == 0;
      const int my_slot = (sg == sg_first) ? 0 : 1;
      const int64_t part = (int64_t)kRows * tp.ntok;  // floats per partial slot
      float* wsp = p.ws + ((int64_t)blockIdx.x * 2 + my_slot) * part;
      for (int c0 = 0; c0 < tp.ntok; c0 += 32) {
        uint32_t v[32];
        if (!dead) {
          tmem_load32(d_taddr + lane_base + (uint32_t)c0, v);
          tmem_load_wait();
        }
        const int nv = tp.ntok - c0 < 32 ? tp.ntok - c0 : 32;  // ntok is a multiple of 16
        if (complete) {
          float a[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) a[i] = __uint_as_float(v[i]);
          store_y_block(tp, &tmap_y, stg, stg_step, a, sc, nv, mtile * tp.ntok + c0, rb, r, tid128, bar);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i < nv) __stcg(wsp + (int64_t)(c0 + i) * kRows + r, __uint_as_float(v[i]));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&d_empty[db]);
      if (!complete) {
        __threadfence();
        named_bar_sync(bar, 128);
        const int64_t i_first = owner_of(seg_begin, p.W, p.G);
        const int64_t i_last = owner_of(seg_begin + T - 1, p.W, p.G);
        const int sf = (range_begin(i_first, p.W, p.G) / T == sg) ? 0 : 1;
        int* ctr = p.cnt + i_first * 2 + sf;
        if (tid128 == 0) {
          const int old = atomicAdd(ctr, 1);
          s_flag[grp] = (old == (int)(i_last - i_first)) ? 1 : 0;
        }
        named_bar_sync(bar, 128);
        if (s_flag[grp]) {
          __threadfence();
          // 32 tokens at a time: each contributor's 32 partials are independent loads
          for (int c0 = 0; c0 < tp.ntok; c0 += 32) {
            float sum[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) sum[i] = 0.f;
            for (int64_t ci = i_first; ci <= i_last; ++ci) {
              const int sl = (range_begin(ci, p.W, p.G) / T == sg) ? 0 : 1;
              const float* src = p.ws + (ci * 2 + sl) * part + (int64_t)c0 * kRows + r;
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (c0 + i < tp.ntok) sum[i] += __ldcg(src + (int64_t)i * kRows);
            }
            const int nv = tp.ntok - c0 < 32 ? tp.ntok - c0 : 32;
            store_y_block(tp, &tmap_y, stg, stg_step, sum, sc, nv, mtile * tp.ntok + c0, rb, r, tid128, bar);
          }
          if (tid128 == 0) atomicExch(ctr, 0);
        }
        named_bar_sync(bar, 128);
      }
    }
  }
  if (tp.y_tma && warp >= kExpWarp0 && ((warp - kExpWarp0) & 3) == 0 && lane == 0) bulk_wait_all();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ host side
int grid_tc(const sp_matrix* h, int64_t W) { return (int)std::min<int64_t>(h->num_sms, W); }

int ntok_for(int64_t M) {
  const int64_t n = std::min<int64_t>(kMaxNtok, (M + 15) / 16 * 16);
  return (int)std::max<int64_t>(16, n);
}

template <int ES, int EG>
sp_status launch_tc_es(const TcParams& tp, const CUtensorMap& map, const CUtensorMap& map_y, size_t smem,
                       cudaStream_t stream, bool pdl) {
  auto kern = linear_tc_kernel<ES, EG>;
  static bool configured[kMaxDevices] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= kMaxDevices) return SP_ERR_UNSUPPORTED;
  if (!configured[dev]) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemLimit) != cudaSuccess) {
      cudaGetLastError();
      return SP_ERR_CUDA;
    }
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)tp.p.G);
  cfg.blockDim = dim3(tc_threads(EG));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, kern, tp, map, map_y) != cudaSuccess) {
    cudaGetLastError();
    return SP_ERR_CUDA;
  }
  return SP_OK;
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::mutex g_encode_mu;

sp_status tensor_map_encoder(PFN_cuTensorMapEncodeTiled_v12000* out) {
  std::lock_guard<std::mutex> lk(g_encode_mu);
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn) {
      cudaGetLastError();
      return SP_ERR_CUDA;
    }
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  *out = g_encode;
  return SP_OK;
}

size_t workspace_bytes_tc(const sp_matrix* h, int64_t M) {
  const int ntok = ntok_for(M);
  const int64_t mt = (M + ntok - 1) / ntok;
  const int64_t W = mt * h->RB * h->T;
  const size_t G = (size_t)grid_tc(h, W);
  return ws_counter_bytes(h->num_sms) + 2 * G * kRows * (size_t)ntok * sizeof(float);
}

sp_status launch_linear_tc(const sp_matrix* h, const uint16_t* x, int64_t M, uint16_t* y, void* ws, size_t ws_bytes,
                           cudaStream_t stream) {
  if (!ws || ws_bytes < workspace_bytes_tc(h, M)) return SP_ERR_WORKSPACE;
  if (M > ((int64_t)1 << 31) / kMaxNtok) return SP_ERR_UNSUPPORTED;
  PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  sp_status st = tensor_map_encoder(&encode);
  if (st != SP_OK) return st;
  TcParams tp{};
  LinearParams& p = tp.p;
  p.buf = h->d_buf;
  p.off = h->d_off;
  p.scale = h->d_scale;
  p.x = x;
  p.y = y;
  p.status = device_status_ptr();
  p.N = h->N;
  p.K = h->K;
  p.T = h->T;
  p.RB = h->RB;
  p.M = (int32_t)M;
  tp.ntok = ntok_for(M);
  tp.mt = (int32_t)((M + tp.ntok - 1) / tp.ntok);
  p.W = (int64_t)tp.mt * h->RB * h->T;
  p.G = grid_tc(h, p.W);
  p.cnt = reinterpret_cast<int*>(ws);
  p.ws = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(ws) + ws_counter_bytes(h->num_sms));
  p.timeout_ns = wait_timeout_ns();
  tmem_split(tp.ntok, &tp.n_a, &tp.n_d, &tp.d_cols);
  tp.a_col0 = (uint32_t)tp.n_d * tp.d_cols;
  tp.b_bytes = (uint32_t)tp.ntok * 128u;
  tp.chunk_off = (tp.b_bytes + 1023u) / 1024u * 1024u;
  p.chunk_region = (uint32_t)((h->max_chunk + 1023) / 1024 * 1024);
  p.slot_bytes = tp.chunk_off + p.chunk_region;
  // base alignment + barriers (3 per slot, D handshakes), TMEM address, flags, and (TMA
  // stores of y) the staging tiles, 1024-byte aligned
  tp.y_tma = (h->N % 8 == 0) ? 1 : 0;
  const size_t ctl_bytes = 8 * (3 * kMaxSlots + kMaxDBufs * (kMaxExpGroups + 1)) + 4 + 4 * kMaxExpGroups + 16;
  // S = slots = A stages in use, a multiple of the expander warpgroups EG: they take items
  // round-robin, so a slot's previous item belongs to the warpgroup now waiting on it, which
  // keeps the parity wait on the slot's full barrier exact.  Three groups where the ring
  // then holds at least two slots per group (token tiles of up to 64 tokens), else two.
  int eg = 0, slots = 0;
  size_t tail = 0;
  for (const int cand : {kMaxExpGroups, 2}) {
    if (cand == kMaxExpGroups && tp.ntok > 64) continue;
    const size_t stg_bytes = tp.y_tma ? (size_t)cand * 2 * kStgBytes : 0;
    const size_t tl = 1024 + (ctl_bytes + 1023) / 1024 * 1024 + stg_bytes;
    if (tl >= kSmemLimit) continue;
    const int sl =
        (int)std::min<size_t>(std::min<size_t>(kMaxSlots, (kSmemLimit - tl) / p.slot_bytes), (size_t)tp.n_a) /
        cand * cand;
    if (sl >= (cand == kMaxExpGroups ? 2 * cand : cand)) {
      eg = cand;
      slots = sl;
      tail = tl;
      break;
    }
  }
  if (eg == 0) return SP_ERR_UNSUPPORTED;
  p.slots = slots;
  tp.stg_off = (uint32_t)((size_t)slots * p.slot_bytes + (ctl_bytes + 1023) / 1024 * 1024);
  // at least 116 KB so that two CTAs never share an SM (each allocates 512 TMEM columns)
  const size_t smem = std::max<size_t>((size_t)slots * p.slot_bytes + tail, 116 * 1024);

  // x [M, K] bf16, box = 64 K-elements x ntok tokens, 128-byte swizzle; rows past M and
  // columns past K read as zero.
  CUtensorMap map;
  const cuuint64_t gdim[2] = {(cuuint64_t)h->K, (cuuint64_t)M};
  const cuuint64_t gstride[1] = {(cuuint64_t)h->K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kTileK, (cuuint32_t)tp.ntok};
  const cuuint32_t estride[2] = {1, 1};
  if (encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(x), gdim, gstride, box, estride,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return SP_ERR_CUDA;
  // y [M, N] bf16 written by TMA stores in boxes of 128 rows x 16 tokens (needs a row pitch
  // that is a multiple of 16 bytes); otherwise the epilogue stores scalars
  CUtensorMap map_y;
  memset(&map_y, 0, sizeof(map_y));
  if (tp.y_tma) {
    const cuuint64_t ydim[2] = {(cuuint64_t)h->N, (cuuint64_t)M};
    const cuuint64_t ystride[1] = {(cuuint64_t)h->N * 2};
    const cuuint32_t ybox[2] = {(cuuint32_t)kRows, (cuuint32_t)kStgBox};
    if (encode(&map_y, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, y, ydim, ystride, ybox, estride,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return SP_ERR_CUDA;
  }
  // after an in-place weight update the launch waits for the whole previous grid (no
  // weight copy may start before its writes are visible)
  const bool pdl = !h->weights_written;
  if (eg == kMaxExpGroups)
    st = h->esize == 2 ? launch_tc_es<2, kMaxExpGroups>(tp, map, map_y, smem, stream, pdl)
                       : launch_tc_es<1, kMaxExpGroups>(tp, map, map_y, smem, stream, pdl);
  else
    st = h->esize == 2 ? launch_tc_es<2, 2>(tp, map, map_y, smem, stream, pdl)
                       : launch_tc_es<1, 2>(tp, map, map_y, smem, stream, pdl);
  if (st == SP_OK) h->weights_written = 0;
  return st;
}

}  // namespace sp
