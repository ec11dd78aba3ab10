"""Seeded synthetic inputs shaped like the Llama-2-7B linear layers.

This module is the one piece shared by the CUDA path's tests/bench and by the
CPU oracle's tests: it makes weights, masks, INT8 (q, s) pairs and activations,
and holds none of the sparse-linear arithmetic itself (no compression, no
products).  Everything is NumPy on the host, driven by
``numpy.random.default_rng(SeedSequence([seed, layer, proj, stream]))``.

Stand-ins for what the paper takes from elsewhere (Sec. 2.1, 3.4):
  * SparseGPT masks -> per-row magnitude masks: in each row the n_prune entries
    with the smallest |w| are dropped, ties broken by the lower column first
    (a stable sort on |w|); n_prune = round-half-even(pct * K / 100).
  * Outlier-aware non-uniform masks -> per-row sparsity drawn uniformly within
    +-10 points of the target (clipped to [0, 90]), with 5% of the columns
    (round(0.05 K), drawn once per matrix) never pruned.
  * GPTQ/SmoothQuant INT8 -> symmetric absmax per output row over the kept
    weights: s = max|w| / 127 (s = 1 for an empty or all-zero row),
    q = clamp(round-half-even(w / s), -127, 127) at kept positions, 0 elsewhere.
"""
from __future__ import annotations

import numpy as np

# The four fused Llama-2-7B linear shapes (N = out features, K = in features).
LLAMA2_7B_SHAPES = {
    "qkv": (12288, 4096),
    "o": (4096, 4096),
    "gate_up": (22016, 4096),
    "down": (4096, 11008),
}
PROJ_IDS = {"qkv": 0, "o": 1, "gate_up": 2, "down": 3, "q": 4}
STREAM_W, STREAM_MASK, STREAM_X, STREAM_RESID = 0, 1, 2, 3


def rng(seed: int, layer: int, proj: int, stream: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([seed, layer, proj, stream]))


def bf16_from_f32(a: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even.  Finite inputs
    (the largest finite pattern plus the rounding bias still fits in 32 bits)."""
    u = np.array(a, dtype=np.float32, copy=True).view(np.uint32)
    lsb = (u >> 16) & 1
    u += 0x7FFF
    u += lsb
    u >>= 16
    return u.astype(np.uint16)


def bf16_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def round_half_even_div(num: int, den: int) -> int:
    q, r = divmod(num, den)
    if 2 * r > den or (2 * r == den and q % 2 == 1):
        q += 1
    return q


def n_pruned(pct: int, K: int) -> int:
    """Entries dropped per row at an integer sparsity percentage."""
    return round_half_even_div(pct * K, 100)


def _normal_bf16(shape, g: np.random.Generator, std: float | None) -> np.ndarray:
    """bf16 bits of std * N(0, 1) (or N(0, 1)), drawn row-chunk by row-chunk; the
    generator's stream is the same as one draw of the full shape."""
    N, K = shape
    out = np.empty((N, K), dtype=np.uint16)
    rows = max(1, (1 << 22) // max(K, 1))
    buf = np.empty((rows, K), dtype=np.float32)
    for r0 in range(0, N, rows):
        r1 = min(N, r0 + rows)
        b = buf[: r1 - r0]
        g.standard_normal(out=b, dtype=np.float32)
        if std is not None:
            b *= np.float32(std)
        out[r0:r1] = bf16_from_f32(b)
    return out


def weight(N: int, K: int, g: np.random.Generator, std: float = 0.02) -> np.ndarray:
    """bf16 bits of W ~ N(0, std^2), shape [N, K]."""
    return _normal_bf16((N, K), g, std)


def activations(M: int, K: int, g: np.random.Generator) -> np.ndarray:
    """bf16 bits of x ~ N(0, 1), shape [M, K]."""
    return _normal_bf16((M, K), g, None)


def _prune_smallest(W: np.ndarray, n_prune_per_row: np.ndarray, keep_cols=None) -> np.ndarray:
    """Keep-mask dropping, per row, the n smallest |w| with ties broken by the lower
    column.  Every entry gets the unique key (|w| bit pattern, column): for
    non-negative floats the bit pattern orders like the value, so the n smallest
    keys are exactly the first n entries of a stable sort on |w|."""
    N, K = W.shape
    assert K < (1 << 20)
    W = np.ascontiguousarray(W, dtype=np.uint16)
    n_prune_per_row = np.asarray(n_prune_per_row, dtype=np.int64)
    cols = np.arange(K, dtype=np.uint64)[None, :]
    if keep_cols is not None:
        cols = cols.copy()
        cols[:, keep_cols] |= np.uint64(1) << np.uint64(40)  # after every prunable column
    mask = np.ones((N, K), dtype=np.uint8)
    rows_per = max(1, (1 << 21) // K)
    key = np.empty((rows_per, K), dtype=np.uint64)
    for r0 in range(0, N, rows_per):
        r1 = min(N, r0 + rows_per)
        kk = key[: r1 - r0]
        np.bitwise_and(W[r0:r1], np.uint16(0x7FFF), out=kk, casting="unsafe")
        kk <<= np.uint64(20)
        kk |= cols
        npr = n_prune_per_row[r0:r1]
        for n in np.unique(npr):
            if n <= 0:
                continue
            sel = np.nonzero(npr == n)[0]
            if n >= K:
                mask[r0 + sel] = 0
                continue
            sub = kk if sel.size == kk.shape[0] else kk[sel]
            thr = np.partition(sub, n - 1, axis=1)[:, n - 1]
            mask[r0 + sel] = sub > thr[:, None]
    return mask


def magnitude_mask(W: np.ndarray, pct: int) -> np.ndarray:
    """uint8 keep-mask [N, K]: per row, drop the n_pruned(pct, K) smallest |w|."""
    N, K = W.shape
    n = np.full(N, n_pruned(pct, K), dtype=np.int64)
    return _prune_smallest(W, n)


def nonuniform_mask(W: np.ndarray, pct: int, g: np.random.Generator):
    """Non-uniform per-row magnitude mask with dense outlier columns.

    Returns (mask, n_prune_per_row, outlier_cols)."""
    N, K = W.shape
    n_out = round_half_even_div(5 * K, 100)
    outliers = np.sort(g.choice(K, size=n_out, replace=False))
    s_row = np.clip(g.uniform(pct - 10.0, pct + 10.0, size=N), 0.0, 90.0)
    n_prune = np.rint(s_row * K / 100.0).astype(np.int64)
    n_prune = np.minimum(np.maximum(n_prune, 0), K - n_out)
    if pct == 0:
        n_prune[:] = 0
    return _prune_smallest(W, n_prune, outliers), n_prune, outliers


def quantize_int8(W: np.ndarray, mask: np.ndarray):
    """(q int8 [N, K], s float32 [N]) by symmetric absmax over the kept weights (row blocks
    at a time; every element's arithmetic is the same as on the whole matrix)."""
    N, K = W.shape
    q = np.empty((N, K), dtype=np.int8)
    s = np.empty(N, dtype=np.float32)
    rows = max(1, (1 << 18) // max(K, 1))
    for r0 in range(0, N, rows):
        r1 = min(N, r0 + rows)
        keep = mask[r0:r1] != 0
        w = bf16_to_f32(W[r0:r1]).astype(np.float64) * keep
        amax = np.abs(w).max(axis=1)
        sr = np.where(amax > 0, amax / 127.0, 1.0).astype(np.float32)
        qq = np.clip(np.rint(w / sr.astype(np.float64)[:, None]), -127, 127).astype(np.int8)
        qq[~keep] = 0
        q[r0:r1] = qq
        s[r0:r1] = sr
    return q, s


def quantize_activations_int8(x: np.ndarray):
    """(qx int8 [M, K], sx float32 [M]) by symmetric absmax per token (row of x, bf16 bits):
    sx = max|x_m| / 127 (1 for an all-zero row), qx = clamp(rne(x / sx), -127, 127)."""
    xf = bf16_to_f32(x).astype(np.float64)
    amax = np.abs(xf).max(axis=1)
    sx = np.where(amax > 0, amax / 127.0, 1.0).astype(np.float32)
    qx = np.clip(np.rint(xf / sx.astype(np.float64)[:, None]), -127, 127).astype(np.int8)
    return qx, sx


# The four fused linears of one Llama-2-7B layer, in the order a decode step runs them.
STACK_SHAPES = ("qkv", "o", "gate_up", "down")


def stack_layer(pct, int8: bool, seed: int = 0, layer: int = 0, std: float = 0.02) -> dict:
    """Seeded host inputs of one layer of the linear stack: {shape: (values, mask, scale or
    None)} with W ~ N(0, std^2) drawn from rng(seed, layer, proj, STREAM_W), per-row magnitude
    masks at `pct` percent (one int for every shape, or {shape: pct}), and for INT8 the
    absmax (q, s) pair."""
    out = {}
    for name in STACK_SHAPES:
        N, K = LLAMA2_7B_SHAPES[name]
        W = weight(N, K, rng(seed, layer, PROJ_IDS[name], STREAM_W), std=std)
        mask = magnitude_mask(W, pct[name] if isinstance(pct, dict) else pct)
        if int8:
            q, s = quantize_int8(W, mask)
            out[name] = (q, mask, s)
        else:
            out[name] = (W, mask, None)
    return out


def layer_sparsity_profile(layers: int, mean: int = 70, spread: int = 10, seed: int = 0) -> list:
    """A per-layer sparsity profile (percent per layer) standing in for an outlier-weighted
    layerwise profile: five levels mean - spread, mean - spread/2, mean, mean + spread/2,
    mean + spread in counts symmetric about the mean (so the profile's mean is exactly
    `mean`), assigned to layers by a seeded permutation."""
    lv = [mean - spread, mean - spread // 2, mean, mean + spread // 2, mean + spread]
    edge = layers // 8
    half = (layers - 2 * edge) // 2 - (layers - 2 * edge) // 6
    mid = layers - 2 * edge - 2 * half
    counts = [edge, half, mid, half, edge]
    prof = [v for v, c in zip(lv, counts) for _ in range(c)]
    order = rng(seed, 0, 11, STREAM_MASK).permutation(layers)
    return [int(prof[i]) for i in order]


def layer_inputs(shape_name: str, pct: int, M: int, seed: int = 0, layer: int = 0):
    """(W, mask, x) for one Llama-2-7B linear at a uniform per-row sparsity."""
    N, K = LLAMA2_7B_SHAPES[shape_name]
    p = PROJ_IDS[shape_name]
    W = weight(N, K, rng(seed, layer, p, STREAM_W))
    mask = magnitude_mask(W, pct)
    x = activations(M, K, rng(seed, layer, p, STREAM_X))
    return W, mask, x
