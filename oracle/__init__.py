"""CPU oracle for the bitmask-compressed sparse linear (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline and
``--impl reference`` legs may import this package.  The product library never
does, and this package never imports the product package: the two share no code.

The arithmetic lives in ``sp_oracle.c`` (plain C, float64); this module only
compiles it (``build()``) and marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sp_oracle.c")
_LIB = os.path.join(_HERE, "libsp_oracle.so")
_lock = threading.Lock()
_lib = None

TILE_K = 64
CHUNK_ROWS = 128
MASK_BYTES = CHUNK_ROWS * 8


def build(force: bool = False) -> str:
    """Compile sp_oracle.c into libsp_oracle.so next to it (gcc, -O2, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _bind(lib):
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    lib.or_geometry.argtypes = [I64, I64, P, P]
    lib.or_compressed_size.argtypes = [P, I64, I64, ctypes.c_int, P]
    lib.or_compressed_size.restype = I64
    lib.or_compress.argtypes = [P, P, I64, I64, ctypes.c_int, P, I64, P]
    lib.or_compress.restype = ctypes.c_int
    lib.or_decompress.argtypes = [P, P, I64, I64, ctypes.c_int, P]
    lib.or_decompress.restype = ctypes.c_int
    lib.or_linear_bf16.argtypes = [P, I64, P, P, I64, I64, P]
    lib.or_linear_int8.argtypes = [P, I64, P, P, P, I64, I64, P]
    lib.or_linear_from_format.argtypes = [P, P, I64, I64, ctypes.c_int, P, P, I64, P]
    lib.or_linear_from_format.restype = ctypes.c_int
    lib.or_residual_add.argtypes = [P, P, P, I64, I64, P]
    lib.or_mul_halves.argtypes = [P, I64, I64, P]
    lib.or_linear_w8a8.argtypes = [P, P, I64, P, P, P, I64, I64, P, P]
    lib.or_masked_update_bf16.argtypes = [P, P, I64, I64, P, ctypes.c_float]
    lib.or_masked_update_bf16.restype = ctypes.c_int
    lib.or_block_encode.argtypes = [P, ctypes.c_int, P, P]
    lib.or_block_encode.restype = ctypes.c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
    return _lib


def use_library(path: str | None):
    """Point this module at another build of sp_oracle.c (the mutation tests build
    deliberately broken copies); None restores the default build."""
    global _lib
    with _lock:
        _lib = None if path is None else _bind(ctypes.CDLL(path))


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def geometry(N: int, K: int) -> tuple[int, int]:
    """(T, RB): number of 64-wide K-tiles and of 128-row blocks."""
    return (K + TILE_K - 1) // TILE_K, (N + CHUNK_ROWS - 1) // CHUNK_ROWS


def compress(W: np.ndarray, mask: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Compressed bytes and chunk offsets of W o mask.  W is uint16 (bf16 bits) or int8."""
    W = np.ascontiguousarray(W)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    N, K = W.shape
    esize = W.dtype.itemsize
    assert esize in (1, 2) and mask.shape == (N, K)
    T, RB = geometry(N, K)
    off = np.zeros(RB * T + 1, dtype=np.uint64)
    lib = _load()
    total = lib.or_compressed_size(_p(mask), N, K, esize, _p(off))
    buf = np.zeros(max(total, 16), dtype=np.uint8)
    rc = lib.or_compress(_p(W), _p(mask), N, K, esize, _p(buf), total, _p(off))
    assert rc == 0
    return buf[:total], off


def decompress(buf: np.ndarray, off: np.ndarray, N: int, K: int, dtype) -> np.ndarray:
    dtype = np.dtype(dtype)
    out = np.zeros((N, K), dtype=dtype)
    buf = np.ascontiguousarray(buf, dtype=np.uint8)
    off = np.ascontiguousarray(off, dtype=np.uint64)
    rc = _load().or_decompress(_p(buf), _p(off), N, K, dtype.itemsize, _p(out))
    if rc != 0:
        raise ValueError("malformed compressed buffer")
    return out


def linear_bf16(x: np.ndarray, W: np.ndarray, mask: np.ndarray) -> np.ndarray:
    """float64 y[M, N] = x . (W o mask)^T from bf16 bit patterns (uint16)."""
    x = np.ascontiguousarray(x, dtype=np.uint16)
    W = np.ascontiguousarray(W, dtype=np.uint16)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    M, K = x.shape
    N = W.shape[0]
    y = np.zeros((M, N), dtype=np.float64)
    _load().or_linear_bf16(_p(x), M, _p(W), _p(mask), N, K, _p(y))
    return y


def linear_int8(x: np.ndarray, q: np.ndarray, mask: np.ndarray, s: np.ndarray) -> np.ndarray:
    """float64 y[M, N] = x . ((q * s[:, None]) o mask)^T."""
    x = np.ascontiguousarray(x, dtype=np.uint16)
    q = np.ascontiguousarray(q, dtype=np.int8)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    s = np.ascontiguousarray(s, dtype=np.float32)
    M, K = x.shape
    N = q.shape[0]
    y = np.zeros((M, N), dtype=np.float64)
    _load().or_linear_int8(_p(x), M, _p(q), _p(mask), _p(s), N, K, _p(y))
    return y


def linear_w8a8(qx: np.ndarray, sx: np.ndarray, qw: np.ndarray, mask: np.ndarray, sw: np.ndarray):
    """INT8 weights and activations: (int64 acc [M, N], float64 y = sx[m] * sw[n] * acc)."""
    qx = np.ascontiguousarray(qx, dtype=np.int8)
    sx = np.ascontiguousarray(sx, dtype=np.float32)
    qw = np.ascontiguousarray(qw, dtype=np.int8)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    sw = np.ascontiguousarray(sw, dtype=np.float32)
    M, K = qx.shape
    N = qw.shape[0]
    assert qw.shape == (N, K) and mask.shape == (N, K) and sx.shape == (M,) and sw.shape == (N,)
    acc = np.zeros((M, N), dtype=np.int64)
    y = np.zeros((M, N), dtype=np.float64)
    _load().or_linear_w8a8(_p(qx), _p(sx), M, _p(qw), _p(mask), _p(sw), N, K, _p(acc), _p(y))
    return acc, y


def linear_from_format(buf, off, N: int, K: int, esize: int, x: np.ndarray, scale=None) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.uint16)
    buf = np.ascontiguousarray(buf, dtype=np.uint8)
    off = np.ascontiguousarray(off, dtype=np.uint64)
    M = x.shape[0]
    y = np.zeros((M, N), dtype=np.float64)
    sp = None
    if scale is not None:
        scale = np.ascontiguousarray(scale, dtype=np.float32)
        sp = _p(scale)
    rc = _load().or_linear_from_format(_p(buf), _p(off), N, K, esize, sp, _p(x), M, _p(y))
    if rc != 0:
        raise ValueError("malformed compressed buffer")
    return y


def block_encode(elems) -> tuple[list[int], int]:
    """Bitmask encoding of one block given in compute-read order: (values, mask)."""
    e = np.ascontiguousarray(np.asarray(elems, dtype=np.int16))
    assert e.size <= 64
    vals = np.zeros(64, dtype=np.int16)
    m = np.zeros(1, dtype=np.uint64)
    c = _load().or_block_encode(_p(e), int(e.size), _p(vals), _p(m))
    return [int(v) for v in vals[:c]], int(m[0])


def residual_add(h: np.ndarray, a: np.ndarray, r: np.ndarray) -> np.ndarray:
    """float64 h + a + r (bf16 inputs, r broadcast over rows), before rounding."""
    h = np.ascontiguousarray(h, dtype=np.uint16)
    a = np.ascontiguousarray(a, dtype=np.uint16)
    r = np.ascontiguousarray(r, dtype=np.uint16)
    M, N = h.shape
    out = np.zeros((M, N), dtype=np.float64)
    _load().or_residual_add(_p(h), _p(a), _p(r), M, N, _p(out))
    return out


def mul_halves(g: np.ndarray) -> np.ndarray:
    """float64 g[:, :F] * g[:, F:] (bf16 input), before rounding."""
    g = np.ascontiguousarray(g, dtype=np.uint16)
    M, F2 = g.shape
    out = np.zeros((M, F2 // 2), dtype=np.float64)
    _load().or_mul_halves(_p(g), M, F2 // 2, _p(out))
    return out


def masked_update_bf16(buf: np.ndarray, off: np.ndarray, N: int, K: int, grad: np.ndarray, lr: float) -> np.ndarray:
    """Algorithm 1's masked step on a compressed bf16 matrix: a copy of `buf` with every
    kept value w replaced by bf16_rne(fmaf(-lr, grad, w)); grad is dense [N, K] float32."""
    out = np.array(buf, dtype=np.uint8, copy=True)
    off = np.ascontiguousarray(off, dtype=np.uint64)
    g = np.ascontiguousarray(grad, dtype=np.float32)
    assert g.shape == (N, K)
    rc = _load().or_masked_update_bf16(_p(out), _p(off), N, K, _p(g), ctypes.c_float(lr))
    if rc != 0:
        raise ValueError("malformed compressed matrix")
    return out
