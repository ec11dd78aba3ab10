/*
 * sp_oracle.c -- plain, slow CPU oracle for the bitmask-compressed sparse linear.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or call
 * this file; only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
 * --impl reference legs use it.  It shares no code, header, table or constant
 * with the CUDA library: the byte layout below is re-derived here from the
 * format description, on its own.
 *
 * What it computes, and where the paper defines it
 * ------------------------------------------------
 *  - Bitmask encoding of a block (Sec. 2.4.1, the 2x8 int16 example): the
 *    nonzeros of a block are kept densely, in the order the compute reads the
 *    block, and one bit per element records which positions are kept.
 *    or_block_encode() is that encoding for any element order.
 *  - The compressed matrix (Sec. 2.4.2): the weight is cut into submatrices,
 *    each stored as dense nonzero values plus a bitmask.  Here a submatrix is a
 *    "chunk": 128 consecutive rows x one 64-wide K-tile.  Chunk layout, in
 *    bytes, little-endian:
 *        [0, 1024)   128 x uint64 masks, one per row of the chunk; bit j (LSB=0)
 *                    of the mask of row r is set iff column 64*t + j of row
 *                    128*rb + r is kept.  Rows >= N and columns >= K are 0.
 *        [1024, ..)  the kept values of row 0, then row 1, ... row 127, each row
 *                    in ascending column order, esize bytes per value
 *                    (bf16 bit pattern: 2 bytes; int8: 1 byte).
 *        padding     zero bytes up to the next multiple of 16.
 *    Chunks are stored row-block major: chunk (rb, t) is number c = rb*T + t,
 *    and starts at byte off[c]; off[0] = 0 and off[RB*T] = total bytes.
 *  - The sparse product (Sec. 2.4.2: tensor cores compute on the decompressed
 *    submatrix, "equivalent to dense"): y = x . (W o Mask)^T, written out as
 *    the definition, in float64, summing over k in ascending order.
 *  - INT8 weights with one fp32 scale per output row (Sec. 3.4 uses INT8
 *    weights): the weight of row n is q[n,k] * s[n]; the oracle multiplies
 *    with exactly those quantized weights.
 *
 *  - INT8 weights and INT8 activations (Sec. 3.4: the quantized sparse models
 *    run with INT8 weights and activations): with per-token activation scales
 *    sx[m] and per-row weight scales sw[n], y[m,n] = sx[m] * sw[n] *
 *    sum_k qx[m,k] * qw[n,k] * Mask[n,k]; the integer sum is exact (int64).
 *  - The masked weight update of sparse training (Sec. 2.1, Algorithm 1): the
 *    gradient is multiplied by the fixed mask, the weights take one step of
 *    size eta, and are multiplied by the mask again, so a pruned weight stays
 *    zero.  On the compressed form only the kept entries exist, so the step
 *    touches exactly the stored values; or_masked_update_bf16() applies it there.
 *
 * Floating point: bf16 -> float32 -> double is exact; bf16 x bf16 and
 * bf16 x (int8 * fp32) products are exact in double; only the k-sum rounds.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_TILE_K 64        /* columns per K-tile, one uint64 mask per row */
#define OR_CHUNK_ROWS 128   /* rows per chunk */
#define OR_MASK_BYTES (OR_CHUNK_ROWS * 8)
#define OR_ALIGN 16

static double or_bf16_to_double(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static int64_t or_ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

static int64_t or_pad16(int64_t b) { return (b + OR_ALIGN - 1) / OR_ALIGN * OR_ALIGN; }

/* Number of K-tiles and row-blocks of an N x K matrix. */
void or_geometry(int64_t N, int64_t K, int64_t* T, int64_t* RB) {
  *T = or_ceil_div(K, OR_TILE_K);
  *RB = or_ceil_div(N, OR_CHUNK_ROWS);
}

/* Mask of row n in K-tile t, read from the dense uint8 mask (nonzero = kept). */
static uint64_t or_row_tile_mask(const uint8_t* mask, int64_t N, int64_t K, int64_t n, int64_t t) {
  uint64_t m = 0;
  if (n >= N) return 0;
  for (int j = 0; j < OR_TILE_K; ++j) {
    int64_t k = t * OR_TILE_K + j;
    if (k < K && mask[n * K + k]) m |= (uint64_t)1 << j;
  }
  return m;
}

static int or_popcount64(uint64_t m) {
  int c = 0;
  while (m) { c += (int)(m & 1u); m >>= 1; }
  return c;
}

/* Fills off[0..RB*T] with chunk byte offsets; returns the total byte count. */
int64_t or_compressed_size(const uint8_t* mask, int64_t N, int64_t K, int esize, uint64_t* off) {
  int64_t T, RB;
  or_geometry(N, K, &T, &RB);
  int64_t pos = 0;
  for (int64_t rb = 0; rb < RB; ++rb) {
    for (int64_t t = 0; t < T; ++t) {
      int64_t kept = 0;
      for (int r = 0; r < OR_CHUNK_ROWS; ++r)
        kept += or_popcount64(or_row_tile_mask(mask, N, K, rb * OR_CHUNK_ROWS + r, t));
      off[rb * T + t] = (uint64_t)pos;
      pos += or_pad16(OR_MASK_BYTES + kept * esize);
    }
  }
  off[RB * T] = (uint64_t)pos;
  return pos;
}

/* Writes the compressed form of W o Mask into out (cap bytes).  W holds esize-byte
 * elements (bf16 bit patterns or int8), row-major [N, K].  Returns 0, or -1 if cap
 * is too small. */
int or_compress(const void* W, const uint8_t* mask, int64_t N, int64_t K, int esize,
                uint8_t* out, int64_t cap, uint64_t* off) {
  int64_t T, RB;
  or_geometry(N, K, &T, &RB);
  int64_t total = or_compressed_size(mask, N, K, esize, off);
  if (total > cap) return -1;
  memset(out, 0, (size_t)total);
  const uint8_t* Wb = (const uint8_t*)W;
  for (int64_t rb = 0; rb < RB; ++rb) {
    for (int64_t t = 0; t < T; ++t) {
      uint8_t* chunk = out + off[rb * T + t];
      uint8_t* vals = chunk + OR_MASK_BYTES;
      int64_t v = 0;
      for (int r = 0; r < OR_CHUNK_ROWS; ++r) {
        int64_t n = rb * OR_CHUNK_ROWS + r;
        uint64_t m = or_row_tile_mask(mask, N, K, n, t);
        for (int b = 0; b < 8; ++b) chunk[r * 8 + b] = (uint8_t)(m >> (8 * b));
        for (int j = 0; j < OR_TILE_K; ++j) {
          if (!((m >> j) & 1u)) continue;
          int64_t k = t * OR_TILE_K + j;
          memcpy(vals + v * esize, Wb + (n * K + k) * esize, (size_t)esize);
          ++v;
        }
      }
    }
  }
  return 0;
}

static uint64_t or_read_u64le(const uint8_t* p) {
  uint64_t m = 0;
  for (int b = 0; b < 8; ++b) m |= (uint64_t)p[b] << (8 * b);
  return m;
}

/* Inverse of or_compress: dense [N, K] of esize-byte elements, zero where masked out. */
int or_decompress(const uint8_t* buf, const uint64_t* off, int64_t N, int64_t K, int esize, void* W_out) {
  int64_t T, RB;
  or_geometry(N, K, &T, &RB);
  uint8_t* Wb = (uint8_t*)W_out;
  memset(Wb, 0, (size_t)(N * K * esize));
  for (int64_t rb = 0; rb < RB; ++rb) {
    for (int64_t t = 0; t < T; ++t) {
      const uint8_t* chunk = buf + off[rb * T + t];
      const uint8_t* vals = chunk + OR_MASK_BYTES;
      int64_t v = 0;
      for (int r = 0; r < OR_CHUNK_ROWS; ++r) {
        int64_t n = rb * OR_CHUNK_ROWS + r;
        uint64_t m = or_read_u64le(chunk + r * 8);
        for (int j = 0; j < OR_TILE_K; ++j) {
          if (!((m >> j) & 1u)) continue;
          int64_t k = t * OR_TILE_K + j;
          if (n >= N || k >= K) return -1; /* malformed: bit outside the matrix */
          memcpy(Wb + (n * K + k) * esize, vals + v * esize, (size_t)esize);
          ++v;
        }
      }
    }
  }
  return 0;
}

/* Definition of the bf16 sparse linear: y[m,n] = sum_k x[m,k] * W[n,k] * Mask[n,k],
 * k ascending, float64.  x [M,K] bf16, W [N,K] bf16, mask [N,K] uint8, y [M,N]. */
void or_linear_bf16(const uint16_t* x, int64_t M, const uint16_t* W, const uint8_t* mask,
                    int64_t N, int64_t K, double* y) {
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t m = 0; m < M; ++m) {
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k)
        if (mask[n * K + k]) acc += or_bf16_to_double(x[m * K + k]) * or_bf16_to_double(W[n * K + k]);
      y[m * N + n] = acc;
    }
  }
}

/* INT8 weights and activations: acc[m,n] = sum_k qx[m,k] * qw[n,k] * Mask[n,k] exactly in
 * int64, then y[m,n] = (sx[m] * sw[n]) * acc in float64 (the scale product is exact). */
void or_linear_w8a8(const int8_t* qx, const float* sx, int64_t M, const int8_t* qw, const uint8_t* mask,
                    const float* sw, int64_t N, int64_t K, int64_t* acc_out, double* y) {
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t m = 0; m < M; ++m) {
      int64_t acc = 0;
      for (int64_t k = 0; k < K; ++k)
        if (mask[n * K + k]) acc += (int64_t)qx[m * K + k] * (int64_t)qw[n * K + k];
      if (acc_out) acc_out[m * N + n] = acc;
      y[m * N + n] = ((double)sx[m] * (double)sw[n]) * (double)acc;
    }
  }
}

/* INT8 weights: y[m,n] = sum_k x[m,k] * (q[n,k] * s[n]) * Mask[n,k], float64. */
void or_linear_int8(const uint16_t* x, int64_t M, const int8_t* q, const uint8_t* mask, const float* s,
                    int64_t N, int64_t K, double* y) {
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    double sn = (double)s[n];
    for (int64_t m = 0; m < M; ++m) {
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k)
        if (mask[n * K + k]) acc += or_bf16_to_double(x[m * K + k]) * ((double)q[n * K + k] * sn);
      y[m * N + n] = acc;
    }
  }
}

/* The same product, read from the compressed bytes instead of the dense arrays.
 * Walks every chunk's masks and packed values in storage order and adds each
 * kept product into y[m, n] in ascending k (tiles are visited in ascending t
 * for each row block, so k ascends per output).  scale may be NULL for bf16. */
int or_linear_from_format(const uint8_t* buf, const uint64_t* off, int64_t N, int64_t K, int esize,
                          const float* scale, const uint16_t* x, int64_t M, double* y) {
  int64_t T, RB;
  or_geometry(N, K, &T, &RB);
  for (int64_t i = 0; i < M * N; ++i) y[i] = 0.0;
  for (int64_t rb = 0; rb < RB; ++rb) {
    for (int64_t t = 0; t < T; ++t) {
      const uint8_t* chunk = buf + off[rb * T + t];
      const uint8_t* vals = chunk + OR_MASK_BYTES;
      int64_t v = 0;
      for (int r = 0; r < OR_CHUNK_ROWS; ++r) {
        int64_t n = rb * OR_CHUNK_ROWS + r;
        uint64_t msk = or_read_u64le(chunk + r * 8);
        for (int j = 0; j < OR_TILE_K; ++j) {
          if (!((msk >> j) & 1u)) continue;
          int64_t k = t * OR_TILE_K + j;
          if (n >= N || k >= K) return -1;
          double w;
          if (esize == 2) {
            uint16_t h = (uint16_t)(vals[2 * v] | (vals[2 * v + 1] << 8));
            w = or_bf16_to_double(h);
          } else {
            w = (double)(int8_t)vals[v] * (double)scale[n];
          }
          ++v;
          for (int64_t m = 0; m < M; ++m) y[m * N + n] += or_bf16_to_double(x[m * K + k]) * w;
        }
      }
    }
  }
  return 0;
}

/* Generic bitmask encoding of one block (Sec. 2.4.1): elems[0..n) are the block's
 * elements listed in the order the compute reads them (the "register layout").
 * Writes the nonzero elements, in that order, to values and returns their count;
 * *mask gets bit i (LSB = 0) set iff elems[i] != 0.  n <= 64. */
int or_block_encode(const int16_t* elems, int n, int16_t* values, uint64_t* mask) {
  int c = 0;
  uint64_t m = 0;
  for (int i = 0; i < n; ++i) {
    if (elems[i] != 0) {
      values[c++] = elems[i];
      m |= (uint64_t)1 << i;
    }
  }
  *mask = m;
  return c;
}

/* Glue of the linear-stack decode step (not part of the paper's method: the benchmark
 * chains the linears of each block with residual adds, no attention or normalisation).
 * Results in float64, before any rounding. */
void or_residual_add(const uint16_t* h, const uint16_t* a, const uint16_t* r, int64_t M, int64_t N, double* out) {
  for (int64_t m = 0; m < M; ++m)
    for (int64_t j = 0; j < N; ++j)
      out[m * N + j] = or_bf16_to_double(h[m * N + j]) + or_bf16_to_double(a[m * N + j]) + or_bf16_to_double(r[j]);
}

void or_mul_halves(const uint16_t* g, int64_t M, int64_t F, double* out) {
  for (int64_t m = 0; m < M; ++m)
    for (int64_t j = 0; j < F; ++j)
      out[m * F + j] = or_bf16_to_double(g[m * 2 * F + j]) * or_bf16_to_double(g[m * 2 * F + F + j]);
}

/* float32 -> bf16 bit pattern, round to nearest, ties to even (finite inputs): add just
 * under half of the dropped 16-bit range, plus one when the kept part is odd, and drop
 * the low half. */
static uint16_t or_float_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

/* The masked update of Algorithm 1 on the compressed form, bf16 values: for every kept
 * (n, k), w[n,k] <- bf16(fmaf(-lr, grad[n,k], w[n,k])), one fused multiply-add in float32
 * and one round to nearest even.  grad is dense [N, K] float32; its masked-out entries are
 * never read.  The masks, offsets and padding do not change.  Updates buf in place;
 * returns 0, or -1 for a mask bit outside the matrix. */
int or_masked_update_bf16(uint8_t* buf, const uint64_t* off, int64_t N, int64_t K, const float* grad, float lr) {
  int64_t T, RB;
  or_geometry(N, K, &T, &RB);
  for (int64_t rb = 0; rb < RB; ++rb) {
    for (int64_t t = 0; t < T; ++t) {
      uint8_t* chunk = buf + off[rb * T + t];
      uint8_t* vals = chunk + OR_MASK_BYTES;
      int64_t v = 0;
      for (int r = 0; r < OR_CHUNK_ROWS; ++r) {
        int64_t n = rb * OR_CHUNK_ROWS + r;
        uint64_t m = or_read_u64le(chunk + r * 8);
        for (int j = 0; j < OR_TILE_K; ++j) {
          if (!((m >> j) & 1u)) continue;
          int64_t k = t * OR_TILE_K + j;
          if (n >= N || k >= K) return -1;
          uint16_t h;
          memcpy(&h, vals + v * 2, 2);
          uint32_t u = (uint32_t)h << 16;
          float w;
          memcpy(&w, &u, sizeof w);
          h = or_float_to_bf16_rne(fmaf(-lr, grad[n * K + k], w));
          memcpy(vals + v * 2, &h, 2);
          ++v;
        }
      }
    }
  }
  return 0;
}
