// sp_cc_common.cuh -- the CUDA-core per-chunk arithmetic shared by the decode kernels
// (sp_linear_cc.cu: one sparse linear per launch; sp_chain.cu: a chain of them in one
// persistent launch): bit-walk helpers, the value streams, the x operand registers and
// the per-row dot product over one chunk row.
#pragma once

#include "sp_internal.cuh"

namespace sp {
namespace cc {
// Index of the most significant set bit, or -1 for 0.
__device__ __forceinline__ int msb32(uint32_t v) {
  int r;
  asm("bfind.u32 %0, %1;" : "=r"(r) : "r"(v));
  return r;
}
// 1 << j for j in [0, 31]; 0 for j = -1 (PTX clamps the shift amount).
__device__ __forceinline__ uint32_t bit32(int j) {
  uint32_t r;
  asm("shl.b32 %0, 1, %1;" : "=r"(r) : "r"(j));
  return r;
}
// acc + a * b with bf16 a, b and an FP32 accumulator (sm_100+ mixed-precision FMA).
__device__ __forceinline__ float fma_bf16(uint16_t a, uint16_t b, float c) {
  float d;
  asm("fma.rn.f32.bf16 %0, %1, %2, %3;" : "=f"(d) : "h"(a), "h"(b), "f"(c));
  return d;
}
__device__ __forceinline__ uint16_t lo16(uint32_t v) { return (uint16_t)(v & 0xffffu); }
__device__ __forceinline__ uint16_t hi16(uint32_t v) { return (uint16_t)(v >> 16); }
// int8 weight -> bf16 bits, exact for |q| <= 128: the byte lands in the mantissa of
// 2^23 + 128 + q, the float subtraction leaves q, and q fits bf16's 8-bit significand.
__device__ __forceinline__ uint16_t i8_to_bf16(uint32_t byte) {
  const float f = __uint_as_float(0x4B000000u | (byte ^ 0x80u)) - 8388736.0f;
  return (uint16_t)(__float_as_uint(f) >> 16);
}

__device__ __forceinline__ uint32_t lds32(uint32_t saddr) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(saddr));
  return v;
}
// Low 32 bits of ({hi, lo} >> n), n clamped to 32.
__device__ __forceinline__ uint32_t funnel_r(uint32_t lo, uint32_t hi, uint32_t n) {
  uint32_t r;
  asm("shf.r.clamp.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(lo), "r"(hi), "r"(n));
  return r;
}
// Clear bit j (no-op for j = -1).
__device__ __forceinline__ uint32_t clear_bit(uint32_t v, int j) { return v & ~bit32(j); }

// One chain's value stream, walked from its highest-column value downward.  The values
// are bf16 halves at byte address `top` (the highest) and below; every second step
// loads one aligned 32-bit word, and a funnel shift realigns odd starting positions.
struct Stream16 {
  uint32_t addr;   // byte address of the aligned word holding the next pair's first value
  uint32_t cur;    // that word
  uint32_t shift;  // 16 if the stream starts at a low half (even index), else 32
  __device__ __forceinline__ void init(uint32_t top_byte) {
    addr = top_byte & ~3u;
    cur = lds32(addr);
    shift = (top_byte & 2u) ? 32u : 16u;
  }
  // next two values: first in the high half, second in the low half
  __device__ __forceinline__ uint32_t next_pair() {
    addr -= 4;
    const uint32_t below = lds32(addr);
    const uint32_t w = funnel_r(below, cur, shift);
    cur = below;
    return w;
  }
};

// One chain's int8 value stream, walked from its highest-column value downward, four values
// per aligned 32-bit load: next_quad() returns the next four values with the first in the
// top byte (a funnel shift realigns a start that is not word-aligned), each byte biased by
// +128 (q ^ 0x80), ready for i8_biased_to_f32.  Reads reach at most 4 bytes above the top
// value and, for an exhausted chain, a few words below the row's first value: still inside
// the slot (the chunk's mask area precedes its values).
struct Stream8 {
  uint32_t addr;   // aligned word holding the lowest byte of the next quad
  uint32_t cur;    // the word above it
  uint32_t shift;  // 8 x (offset of the quad's lowest byte in its word)
  __device__ __forceinline__ void init(uint32_t top_byte) {
    const uint32_t low = top_byte - 3u;
    addr = low & ~3u;
    shift = 8u * (low & 3u);
    cur = lds32(addr + 4u);
  }
  __device__ __forceinline__ uint32_t next_quad() {
    const uint32_t below = lds32(addr);
    const uint32_t w = funnel_r(below, cur, shift);
    cur = below;
    addr -= 4u;
    return w ^ 0x80808080u;
  }
};
// Byte i (0..3) of a biased quad as the exact FP32 value q: the byte goes into the low
// mantissa byte of 0x4B000000 (2^23), giving 2^23 + (q + 128), and one subtraction leaves q.
__device__ __forceinline__ float i8_biased_to_f32(uint32_t quad, int i) {
  return __uint_as_float(__byte_perm(quad, 0x4B000000u, 0x7540u | (uint32_t)i)) - 8388736.0f;
}

// acc + a * b in FP32 as one instruction that the compiler predicates under a branch-free
// guard (a plain fmaf there may become an FMA plus a select).
__device__ __forceinline__ float fma_f32_asm(float a, float b, float c) {
  float d;
  asm("fma.rn.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// x of one chunk's K-tile as shuffle sources: lane j holds x[m, 64t+j] (XL) and
// x[m, 64t+32+j] (XH), two batch rows per register.
template <int M>
__device__ __forceinline__ void load_x(const uint8_t* slot, uint32_t chunk_region, int lane,
                                       uint32_t (&XL)[(M + 1) / 2], uint32_t (&XH)[(M + 1) / 2]) {
  const uint16_t* xs = reinterpret_cast<const uint16_t*>(slot + chunk_region);
#pragma unroll
  for (int q = 0; q < (M + 1) / 2; ++q) {
    const uint32_t a0 = xs[(2 * q) * 64 + lane], b0 = xs[(2 * q) * 64 + 32 + lane];
    const uint32_t a1 = (2 * q + 1 < M) ? xs[(2 * q + 1) * 64 + lane] : 0u;
    const uint32_t b1 = (2 * q + 1 < M) ? xs[(2 * q + 1) * 64 + 32 + lane] : 0u;
    XL[q] = a0 | (a1 << 16);
    XH[q] = b0 | (b1 << 16);
  }
}

// acc[m] += sum over the kept columns j of one chunk row of value(j) * x[m, 64t+j].
// The row's 64-bit mask (lo, hi) splits into two 32-column halves walked as two
// independent chains, each from its highest set bit down (bfind), consuming that
// half's values from the top; the x operand comes by shuffle from lane j % 32.  `e0`
// is the index of the row's first value in the chunk's packed values; plo / pc are the
// kept counts of the low half / the row.  Every lane of the warp calls this together.
template <int M, int ES>
__device__ __forceinline__ void row_dot(uint32_t lo, uint32_t hi, int plo, int pc, int e0, const uint8_t* vals,
                                        const uint32_t (&XL)[(M + 1) / 2], const uint32_t (&XH)[(M + 1) / 2],
                                        float (&acc)[M]) {
  constexpr int MP = (M + 1) / 2;
  const int top_lo = e0 + plo - 1;  // highest-column value of the low half
  const int top_hi = e0 + pc - 1;   // ... of the high half
  const int iters = (int)__reduce_max_sync(0xffffffffu, (unsigned)max(plo, pc - plo));
  if constexpr (ES == 2 && M <= 4) {
    // bf16, small batch: two chain steps per loop trip share one word load per chain,
    // and each chain keeps its own accumulators
    float accl[M], acch[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
      accl[m] = 0.f;
      acch[m] = 0.f;
    }
    Stream16 sl, sh;
    const uint32_t vbase = smem_u32(vals);
    sl.init(vbase + 2u * (uint32_t)top_lo);
    sh.init(vbase + 2u * (uint32_t)top_hi);
    for (int q = 0; q < iters; q += 2) {
      const uint32_t wl = sl.next_pair(), wh = sh.next_pair();
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int jl = msb32(lo), jh = msb32(hi);
        lo = clear_bit(lo, jl);
        hi = clear_bit(hi, jh);
        const uint16_t vl = h == 0 ? hi16(wl) : lo16(wl);
        const uint16_t vh = h == 0 ? hi16(wh) : lo16(wh);
#pragma unroll
        for (int r = 0; r < MP; ++r) {
          const uint32_t xl = __shfl_sync(0xffffffffu, XL[r], jl);
          const uint32_t xh = __shfl_sync(0xffffffffu, XH[r], jh);
          if (jl >= 0) {
            accl[2 * r] = fma_bf16(vl, lo16(xl), accl[2 * r]);
            if (2 * r + 1 < M) accl[2 * r + 1] = fma_bf16(vl, hi16(xl), accl[2 * r + 1]);
          }
          if (jh >= 0) {
            acch[2 * r] = fma_bf16(vh, lo16(xh), acch[2 * r]);
            if (2 * r + 1 < M) acch[2 * r + 1] = fma_bf16(vh, hi16(xh), acch[2 * r + 1]);
          }
        }
      }
    }
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] += accl[m] + acch[m];
  } else if constexpr (ES == 1 && M == 1) {
    // int8 values, one batch row: four chain steps per loop trip share one word load per
    // chain (Stream8); each byte becomes its exact FP32 value by a byte permute into the
    // mantissa of 2^23 and one FP32 subtraction (no int -> float conversion on the
    // quarter-rate pipe that the walk's bfind already uses), and x is FP32 in the shuffle
    // registers.  Measured on gate_up: 32.4 -> 29.1 us per launch.
    float accl = 0.f, acch = 0.f;
    const uint32_t xl32 = XL[0] << 16, xh32 = XH[0] << 16;
    Stream8 sl, sh;
    const uint32_t vbase = smem_u32(vals);
    sl.init(vbase + (uint32_t)top_lo);
    sh.init(vbase + (uint32_t)top_hi);
    for (int q = 0; q < iters; q += 4) {
      const uint32_t wl = sl.next_quad(), wh = sh.next_quad();
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const int jl = msb32(lo), jh = msb32(hi);
        lo = clear_bit(lo, jl);
        hi = clear_bit(hi, jh);
        const float vl = i8_biased_to_f32(wl, 3 - h);
        const float vh = i8_biased_to_f32(wh, 3 - h);
        const uint32_t xl = __shfl_sync(0xffffffffu, xl32, jl);
        const uint32_t xh = __shfl_sync(0xffffffffu, xh32, jh);
        if (jl >= 0) accl = fma_f32_asm(vl, __uint_as_float(xl), accl);
        if (jh >= 0) acch = fma_f32_asm(vh, __uint_as_float(xh), acch);
      }
    }
    acc[0] += accl + acch;
  } else if constexpr (ES == 1 && M <= 4) {
    // int8 values, small batch: each chain keeps its own accumulators; a value is one
    // signed byte load and one int -> float conversion, x[m, j] is widened from bf16 by a
    // shift, and the product (int8 x bf16, exact in FP32) is added with an FP32 FMA
    float accl[M], acch[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
      accl[m] = 0.f;
      acch[m] = 0.f;
    }
    const int8_t* v8 = reinterpret_cast<const int8_t*>(vals);
#pragma unroll 2
    for (int q = 0; q < iters; ++q) {
      const int jl = msb32(lo), jh = msb32(hi);
      lo = clear_bit(lo, jl);
      hi = clear_bit(hi, jh);
      // unconditional loads (an exhausted chain reads at most 32 bytes below the row's first
      // value, still inside the chunk's mask area); only the FMAs are predicated
      const float wl = (float)v8[top_lo - q];
      const float wh = (float)v8[top_hi - q];
#pragma unroll
      for (int r = 0; r < MP; ++r) {
        const uint32_t xl = __shfl_sync(0xffffffffu, XL[r], jl);
        const uint32_t xh = __shfl_sync(0xffffffffu, XH[r], jh);
        if (jl >= 0) {
          accl[2 * r] = fmaf(wl, __uint_as_float(xl << 16), accl[2 * r]);
          if (2 * r + 1 < M) accl[2 * r + 1] = fmaf(wl, __uint_as_float(xl & 0xffff0000u), accl[2 * r + 1]);
        }
        if (jh >= 0) {
          acch[2 * r] = fmaf(wh, __uint_as_float(xh << 16), acch[2 * r]);
          if (2 * r + 1 < M) acch[2 * r + 1] = fmaf(wh, __uint_as_float(xh & 0xffff0000u), acch[2 * r + 1]);
        }
      }
    }
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] += accl[m] + acch[m];
  } else {
    // larger batches: one value per chain step, one accumulator set
#pragma unroll 2
    for (int q = 0; q < iters; ++q) {
      const int jl = msb32(lo), jh = msb32(hi);
      lo = clear_bit(lo, jl);
      hi = clear_bit(hi, jh);
      uint16_t wl = 0, wh = 0;
      if (ES == 2) {
        if (jl >= 0) wl = reinterpret_cast<const uint16_t*>(vals)[top_lo - q];
        if (jh >= 0) wh = reinterpret_cast<const uint16_t*>(vals)[top_hi - q];
      } else {
        if (jl >= 0) wl = i8_to_bf16(vals[top_lo - q]);
        if (jh >= 0) wh = i8_to_bf16(vals[top_hi - q]);
      }
#pragma unroll
      for (int r = 0; r < MP; ++r) {
        const uint32_t xl = __shfl_sync(0xffffffffu, XL[r], jl);
        const uint32_t xh = __shfl_sync(0xffffffffu, XH[r], jh);
        if (jl >= 0) {
          acc[2 * r] = fma_bf16(wl, lo16(xl), acc[2 * r]);
          if (2 * r + 1 < M) acc[2 * r + 1] = fma_bf16(wl, hi16(xl), acc[2 * r + 1]);
        }
        if (jh >= 0) {
          acc[2 * r] = fma_bf16(wh, lo16(xh), acc[2 * r]);
          if (2 * r + 1 < M) acc[2 * r + 1] = fma_bf16(wh, hi16(xh), acc[2 * r + 1]);
        }
      }
    }
  }
}

}  // namespace cc
}  // namespace sp
