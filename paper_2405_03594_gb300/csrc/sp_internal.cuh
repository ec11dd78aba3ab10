// sp_internal.cuh -- internals shared by the libsp translation units: the handle,
// kernel parameter blocks, and thin inline-PTX wrappers for sm_103a (mbarrier,
// bulk copies, named barriers, global timer).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/sp.h"

#define SP_MAGIC 0x53504d31u  // "SPM1"

struct sp_matrix {
  uint32_t magic;
  int64_t N, K;
  int32_t T, RB;
  sp_dtype dtype;
  int32_t esize;
  int64_t nnz;
  uint64_t bytes;
  uint64_t max_chunk;
  uint32_t max_quarter;  // most kept entries in one 32-row quarter of a chunk
  uint8_t* d_buf;
  uint64_t* d_off;
  uint64_t* d_qidx;      // per chunk: kept entries before rows 32, 64, 96 and in all 128 rows
                         // (16 bits each, low to high), derived from the masks at compression
  float* d_scale;
  sp_alloc_fn alloc;
  sp_free_fn free_fn;
  void* ctx;
  int32_t device;
  int32_t num_sms;
  // Set by sp_masked_update, which rewrites d_buf in place; cleared by the next linear
  // launch on this handle, which then goes without programmatic dependent launch: the
  // decode kernels copy their first weight chunks before griddepcontrol.wait, and only
  // that wait makes the previous grid's writes visible.
  mutable int32_t weights_written;
};

namespace sp {

constexpr int kTileK = SP_TILE_K;
constexpr int kRows = SP_CHUNK_ROWS;
constexpr int kMaskBytes = SP_CHUNK_MASK_BYTES;

// Work decomposition shared by every sp_linear kernel ("stream-K" over chunks).
// The W = MT * RB * T work items (token tile mt, chunk c = rb*T + t) are cut into G
// contiguous ranges, CTA i taking [i*W/G, (i+1)*W/G).  A (mt, rb) pair whose T
// chunks all fall in one CTA is finished there; otherwise every contributing CTA
// stores a fp32 partial in its slot (0 = its first segment, 1 = its last), and the
// last one to arrive sums the partials in CTA order and writes y.
__host__ __device__ inline int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }
__host__ __device__ inline int64_t range_begin(int64_t i, int64_t W, int64_t G) { return i * W / G; }
__host__ __device__ inline int64_t owner_of(int64_t w, int64_t W, int64_t G) { return ((w + 1) * G - 1) / W; }

struct LinearParams {
  const uint8_t* buf;
  const uint64_t* off;
  const float* scale;   // INT8 only
  const uint16_t* x;    // bf16 bits [M, K]
  uint16_t* y;          // bf16 bits [M, N]
  float* ws;            // partials [2G][kRows][Mt]
  int* cnt;             // arrival counters [2G]
  int* status;
  int64_t N, K;
  int32_t T, RB;
  int32_t M;            // rows of x handled by this launch
  int64_t W;            // work items
  int32_t G;            // CTAs
  int32_t slots;        // ring slots
  uint32_t slot_bytes;  // bytes per ring slot (chunk region + x tile region)
  uint32_t chunk_region;// bytes reserved for the chunk inside a slot
  uint64_t timeout_ns;
  int32_t cluster;      // CUDA-core kernel: > 1 = split each row block over this many CTAs of
                        // one thread-block cluster; <= 1 = stream-K over the workspace
  uint32_t part_off;    // cluster mode: shared-memory offset of the CTA's FP32 partial
  uint32_t comb_off;    // warp-per-chunk kernel: shared-memory offset of the warps' partials
  uint64_t probe_ns;    // 0, except in the failure-path test: consumer warp 0 of CTA 0 first
                        // waits this long on a barrier that nothing completes
  int32_t epi;          // CUDA-core kernels: the output epilogue (sp_chain_epilogue; 0 = store)
  const uint16_t* r;    // SP_EPI_RESIDUAL: bf16 [N] residual vector
};

// Workspace layout, fixed per device so that calls with different grids can share it:
// [arrival counters for up to 2 * kMaxGridPerSm * SMs partial slots][fp32 partials].
// Every call leaves the counters at zero.
constexpr int kMaxGridPerSm = 4;
constexpr int kMaxTokens = 16;  // batch rows per CUDA-core launch (larger batches take several)
inline size_t ws_counter_bytes(int num_sms) {
  return ((size_t)2 * kMaxGridPerSm * num_sms * sizeof(int) + 255) / 256 * 256;
}

enum : int { kStatusOk = 0, kStatusTimeout = 1, kStatusBadFormat = 2 };

// ---------------------------------------------------------------- device helpers
#if defined(__CUDACC__)
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with the given parity.  Returns false once
// `timeout_ns` of global time has passed without completion.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > timeout_ns) return false;
  }
}
// try_wait with a suspend-time hint: the thread sleeps until the phase completes or about
// `hint_ns` pass, instead of returning at once (fewer issue slots spent waiting).
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}
// Bounded wait as mbar_wait, sleeping in the hardware between checks.
__device__ __forceinline__ bool mbar_wait_sleep(uint64_t* bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (true) {
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if (global_ns() - t0 > timeout_ns) return false;
  }
}
// 1-D bulk copy global -> shared, completing `bytes` of transaction on `bar`.
// dst, src and bytes must be multiples of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void bulk_g2s_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                              uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}
// 1-D bulk copy shared -> global in the issuing thread's bulk async-group.  dst, src and
// bytes must be multiples of 16.
__device__ __forceinline__ void bulk_s2g(void* dst, const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_u32(src)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void bulk_wait_read() {  // at most N groups still reading shared memory
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// generic-proxy writes of shared memory become visible to the async proxy (TMA, bulk copies)
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// 2-D TMA tile load into shared memory, completing its bytes on `bar`.  The innermost
// coordinate c0 times the element size must be a multiple of 16 bytes.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// A warp-wide window of 32 consecutive chunk offsets held one per lane, so that a
// producer needs one coalesced global load per 31 chunks instead of a dependent L2
// round trip per chunk.  Every lane of the warp must call at() with the same c.
// Kept entries in chunk rows [0, 32q) -- the rows of the warps before warp quarter q of
// a 128-row chunk: each lane sums its rows lane, lane + 32, ..., then one warp reduction
// (a reduction per quarter would make the last warp of a chunk the slowest).
__device__ __forceinline__ int kept_before_quarter(const uint64_t* masks, int q, int lane) {
  int s = 0;
  for (int k = 0; k < q; ++k) s += __popcll(masks[lane + 32 * k]);
  return (int)__reduce_add_sync(0xffffffffu, (unsigned)s);
}

struct OffsetWindow {
  const uint64_t* off;
  int64_t n_off;  // entries in off[]
  int64_t base;
  uint64_t v;
  __device__ __forceinline__ void refill(int64_t c) {
    base = c;
    const int lane = threadIdx.x & 31;
    v = (c + lane < n_off) ? __ldg(off + c + lane) : 0ull;
  }
  __device__ __forceinline__ void init(const uint64_t* o, int64_t n, int64_t c) {
    off = o;
    n_off = n;
    refill(c);
  }
  // (off[c], off[c + 1])
  __device__ __forceinline__ void at(int64_t c, uint64_t* o0, uint64_t* o1) {
    if (c < base || c + 1 - base >= 32) refill(c);
    *o0 = __shfl_sync(0xffffffffu, v, (int)(c - base));
    *o1 = __shfl_sync(0xffffffffu, v, (int)(c + 1 - base));
  }
};

// Programmatic dependent launch: wait for the preceding grid in the stream (and its
// memory) / allow the next grid to start its prologue.  No-ops without the launch
// attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
// Thread-block cluster helpers (every thread of every CTA of the cluster must take part).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// shared::cta address -> the same offset in CTA `rank` of the cluster (shared::cluster window)
__device__ __forceinline__ uint32_t cluster_map(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ float ld_cluster_f32(uint32_t caddr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(caddr) : "memory");
  return v;
}
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
__device__ __forceinline__ void set_status(int* status, int code) {
  if (status) atomicCAS(status, kStatusOk, code);
}
__device__ __forceinline__ float bf16_bits_to_float(uint32_t h) { return __uint_as_float(h << 16); }
__device__ __forceinline__ uint16_t float_to_bf16_bits_rn(float f) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}
#endif

// ---------------------------------------------------------------- host-side entry points between TUs
sp_status launch_compress(const void* w, const uint8_t* mask, int64_t N, int64_t K, sp_dtype dt, const float* scale,
                          sp_alloc_fn alloc, sp_free_fn free_fn, void* ctx, cudaStream_t stream, sp_matrix** out);
sp_status launch_decompress(const sp_matrix* h, void* w_out, cudaStream_t stream);
// allow_cluster: each launch takes the configuration select_cc picks for its batch rows: a
// thread-block cluster over each row block (no workspace needed) or stream-K with split-K
// partials in the workspace; without it every launch is stream-K.
sp_status launch_linear_cc(const sp_matrix* h, const uint16_t* x, int64_t M, uint16_t* y, void* ws, size_t ws_bytes,
                           cudaStream_t stream, bool allow_cluster = true, uint64_t probe_ns = 0, int32_t epi = 0,
                           const uint16_t* r = nullptr);
size_t workspace_bytes_cc(const sp_matrix* h, int64_t M);
int cc_kernel_kind(const sp_matrix* h, int64_t M);  // 0 thread-per-row, 1 warp-per-chunk, -1 none fits
sp_status launch_linear_tc(const sp_matrix* h, const uint16_t* x, int64_t M, uint16_t* y, void* ws, size_t ws_bytes,
                           cudaStream_t stream);
size_t workspace_bytes_tc(const sp_matrix* h, int64_t M);
sp_status tensor_map_encoder(PFN_cuTensorMapEncodeTiled_v12000* out);  // cuTensorMapEncodeTiled, looked up once
int* device_status_ptr();            // this device's status word (device address)
uint64_t wait_timeout_ns();          // bounded-wait limit for kernels
void* dev_alloc(const sp_matrix* h, size_t bytes);
void dev_free(const sp_matrix* h, void* p);

}  // namespace sp
