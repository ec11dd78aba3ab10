"""Thin ctypes binding of libsp (include/sp.h).  Argument marshalling only: every
step of compression and of the sparse product runs in the library's CUDA kernels.
PyTorch supplies device memory (through the allocator callbacks) and streams.

Importing this module loads libsp.so and raises if it is missing: there is no CPU
or PyTorch fallback for any operation here.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsp.so")

SP_BF16, SP_INT8 = 0, 1
PATHS = {"auto": 0, "cuda_core": 1, "tensor_core": 2}
STATUS = {
    0: "SP_OK", 1: "SP_ERR_INVALID_ARG", 2: "SP_ERR_UNSUPPORTED", 3: "SP_ERR_ALIGNMENT", 4: "SP_ERR_CUDA",
    5: "SP_ERR_OUT_OF_MEMORY", 6: "SP_ERR_TIMEOUT", 7: "SP_ERR_BAD_HANDLE", 8: "SP_ERR_WORKSPACE",
}
SP_ERR_UNSUPPORTED = 2
# every function declared in include/sp.h and include/sp_stack.h
EXPORTS = ["sp_compress", "sp_decompress", "sp_workspace_size", "sp_linear", "sp_linear_ex", "sp_launch_count",
           "sp_linear_noalloc", "sp_test_expired_wait", "sp_masked_update", "sp_linear_w8a8", "sp_w8a8_workspace_size",
           "sp_clone", "sp_free", "sp_info", "sp_copy_out", "sp_check", "sp_status_string",
           "sp_copy_columns", "sp_residual_add", "sp_mul_halves", "sp_mul_pairs", "sp_chain_workspace_size",
           "sp_chain_run", "sp_linear_epi"]


KERNELS = {0: "", 1: "linear_cc_kernel", 2: "linear_ccw_kernel", 3: "linear_tc_kernel"}  # SP_KERNEL_*


class SpError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {STATUS.get(code, code)}")


class SpInfo(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64), ("k", ctypes.c_int64), ("tiles", ctypes.c_int64),
                ("row_blocks", ctypes.c_int64), ("dtype", ctypes.c_int32), ("device", ctypes.c_int32),
                ("nnz", ctypes.c_int64), ("bytes", ctypes.c_uint64), ("max_chunk_bytes", ctypes.c_uint64),
                ("scale_bytes", ctypes.c_uint64)]


EPILOGUES = {"store": 0, "residual": 1, "pair_product": 2}  # sp_chain_epilogue


class SpChainOp(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("x", ctypes.c_void_p), ("ldx", ctypes.c_int64), ("y", ctypes.c_void_p),
                ("ldy", ctypes.c_int64), ("r", ctypes.c_void_p), ("epilogue", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


ALLOC_FN = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)
FREE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p)


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"libsp.so not built at {path}: run __graft_entry__.build() (no fallback exists)")
    lib = ctypes.CDLL(path)
    P, I64, SZ = ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t
    lib.sp_compress.argtypes = [P, P, I64, I64, ctypes.c_int, P, ALLOC_FN, FREE_FN, P, P, ctypes.POINTER(P)]
    lib.sp_decompress.argtypes = [P, P, P]
    lib.sp_workspace_size.argtypes = [P, I64, ctypes.POINTER(SZ)]
    lib.sp_linear.argtypes = [P, P, I64, P, P, SZ, P]
    lib.sp_linear_ex.argtypes = [P, P, I64, P, P, SZ, ctypes.c_int, P]
    lib.sp_launch_count.argtypes = [P, I64, ctypes.c_int, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int32)]
    lib.sp_linear_noalloc.argtypes = [P, P, I64, P, P]
    lib.sp_test_expired_wait.argtypes = [P, P, I64, P, P, SZ, ctypes.c_uint32, P]
    lib.sp_masked_update.argtypes = [P, P, ctypes.c_float, P]
    lib.sp_linear_w8a8.argtypes = [P, P, P, I64, P, P, SZ, P]
    lib.sp_w8a8_workspace_size.argtypes = [P, I64, ctypes.POINTER(SZ)]
    lib.sp_clone.argtypes = [P, ALLOC_FN, FREE_FN, P, P, ctypes.POINTER(P)]
    lib.sp_free.argtypes = [P]
    lib.sp_info.argtypes = [P, ctypes.POINTER(SpInfo)]
    lib.sp_copy_out.argtypes = [P, P, SZ, P, SZ]
    lib.sp_check.argtypes = [P]
    lib.sp_copy_columns.argtypes = [P, P, I64, I64, I64, I64, P]
    lib.sp_residual_add.argtypes = [P, P, P, I64, I64, P]
    lib.sp_mul_halves.argtypes = [P, P, I64, I64, P]
    lib.sp_mul_pairs.argtypes = [P, P, I64, I64, P]
    lib.sp_linear_epi.argtypes = [P, P, I64, P, ctypes.c_int32, P, P, SZ, P]
    lib.sp_chain_workspace_size.argtypes = [I64, ctypes.POINTER(SZ)]
    lib.sp_chain_run.argtypes = [ctypes.POINTER(SpChainOp), ctypes.c_int32, I64, P, SZ, P]
    lib.sp_status_string.argtypes = [ctypes.c_int]
    lib.sp_status_string.restype = ctypes.c_char_p
    for name in EXPORTS:
        if name != "sp_status_string":
            getattr(lib, name).restype = ctypes.c_int
    return lib


_lib = load_library()

# ------------------------------------------------------------------ torch-backed allocator
_live = {}
# re-entrant: a handle collected while this thread holds the lock (its __del__ frees buffers
# through _free) must not deadlock
_live_lock = threading.RLock()


def _alloc(nbytes, ctx):
    try:
        t = torch.empty(int(nbytes), dtype=torch.uint8, device=torch.device("cuda", torch.cuda.current_device()))
    except Exception:
        return None
    p = t.data_ptr()
    with _live_lock:
        _live[p] = t
    return p


def _free(ptr, ctx):
    with _live_lock:
        _live.pop(ptr, None)


_ALLOC = ALLOC_FN(_alloc)
_FREE = FREE_FN(_free)


def _check(code: int, where: str):
    if code != 0:
        raise SpError(code, where)


# The current stream's raw handle without building a torch.cuda.Stream object per call (a
# decode step makes ~130 calls; the public route costs a few microseconds of host time each).
_RAW_STREAM = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(stream=None, device: int | None = None):
    if stream is not None:
        return stream.cuda_stream
    if _RAW_STREAM is not None and device is not None:
        return _RAW_STREAM(device)
    return torch.cuda.current_stream().cuda_stream


def _ptr(t: torch.Tensor | None) -> ctypes.c_void_p:
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


class SparseMatrix:
    """A compressed weight owned by libsp (the handle) with torch-allocated buffers.

    The buffers come from PyTorch's caching allocator on the stream that was current at
    compression, so, as for any torch tensor, their reuse after release is ordered on that
    stream only: work queued on other streams must be complete before the handle is
    dropped (free() synchronises the device first; garbage collection does not)."""

    def __init__(self, handle: ctypes.c_void_p):
        self._h = handle
        info = SpInfo()
        _check(_lib.sp_info(self._h, ctypes.byref(info)), "sp_info")
        self.info = info
        self.n, self.k = int(info.n), int(info.k)
        self.dtype = "int8" if info.dtype == SP_INT8 else "bf16"
        self.device = int(info.device)

    @property
    def handle(self):
        return self._h

    def workspace_size(self, m: int) -> int:
        b = ctypes.c_size_t()
        _check(_lib.sp_workspace_size(self._h, m, ctypes.byref(b)), "sp_workspace_size")
        return int(b.value)

    def launch_count(self, m: int, path: str = "auto") -> int:
        """Kernel launches that linear() makes for a batch of m rows on `path`."""
        n = ctypes.c_int64()
        _check(_lib.sp_launch_count(self._h, m, PATHS[path], ctypes.byref(n), None), "sp_launch_count")
        return int(n.value)

    def kernel_name(self, m: int, path: str = "auto") -> str:
        """Name of the kernel that linear() runs for a batch of m rows on `path`."""
        n, k = ctypes.c_int64(), ctypes.c_int32()
        _check(_lib.sp_launch_count(self._h, m, PATHS[path], ctypes.byref(n), ctypes.byref(k)), "sp_launch_count")
        return KERNELS[k.value]

    def linear(self, x: torch.Tensor, out: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
               path: str = "auto", stream=None) -> torch.Tensor:
        """y = x . (W o Mask)^T with x [m, K] bf16 on this matrix's device."""
        assert x.dtype == torch.bfloat16 and x.dim() == 2 and x.shape[1] == self.k and x.is_contiguous()
        m = x.shape[0]
        if out is None:
            out = torch.empty((m, self.n), dtype=torch.bfloat16, device=x.device)
        if workspace is None:
            workspace = workspace_for(self.workspace_size(m), x.device)
        _check(_lib.sp_linear_ex(self._h, x.data_ptr(), m, out.data_ptr(), workspace.data_ptr(), workspace.numel(),
                                 PATHS[path], _stream(stream, self.device)), "sp_linear")
        return out

    def linear_epi(self, x: torch.Tensor, out: torch.Tensor, epilogue: str, r: torch.Tensor | None = None,
                   workspace: torch.Tensor | None = None, stream=None) -> bool:
        """sp_linear_epi: out = epilogue(x . (W o Mask)^T) with "store", "residual" (out updated
        in place with the bf16 vector r [N]) or "pair_product" (out [m, N/2]).  Returns False,
        launching nothing, where the batch would run on the tensor-core kernel (the caller
        then uses linear() and the glue call)."""
        assert x.dtype == torch.bfloat16 and x.dim() == 2 and x.shape[1] == self.k and x.is_contiguous()
        m = x.shape[0]
        ny = self.n // 2 if epilogue == "pair_product" else self.n
        assert out.dtype == torch.bfloat16 and out.shape == (m, ny) and out.is_contiguous()
        if workspace is None:
            workspace = workspace_for(self.workspace_size(m), x.device)
        code = _lib.sp_linear_epi(self._h, x.data_ptr(), m, out.data_ptr(), EPILOGUES[epilogue],
                                  0 if r is None else r.data_ptr(), workspace.data_ptr(), workspace.numel(),
                                  _stream(stream, self.device))
        if code == SP_ERR_UNSUPPORTED:  # a tensor-core batch
            return False
        _check(code, "sp_linear_epi")
        return True

    def linear_noalloc(self, x: torch.Tensor, out: torch.Tensor, stream=None) -> torch.Tensor:
        """sp_linear_noalloc: the decode kernel with the library's own static scratch, for
        callers that cannot allocate device memory; `out` [m, N] bf16 must be given."""
        assert x.dtype == torch.bfloat16 and x.dim() == 2 and x.shape[1] == self.k and x.is_contiguous()
        assert out.dtype == torch.bfloat16 and out.shape == (x.shape[0], self.n) and out.is_contiguous()
        _check(_lib.sp_linear_noalloc(self._h, _ptr(x), x.shape[0], _ptr(out), _stream(stream, self.device)), "sp_linear_noalloc")
        return out

    def test_expired_wait(self, x: torch.Tensor, out: torch.Tensor, workspace: torch.Tensor, wait_ms: int,
                          stream=None) -> None:
        """sp_test_expired_wait: the decode kernel with one warp's bounded wait made to expire
        (the failure-path test); sp.check() afterwards raises SP_ERR_TIMEOUT."""
        assert x.dtype == torch.bfloat16 and x.dim() == 2 and x.shape[1] == self.k and x.is_contiguous()
        assert out.dtype == torch.bfloat16 and out.shape == (x.shape[0], self.n) and out.is_contiguous()
        _check(_lib.sp_test_expired_wait(self._h, _ptr(x), x.shape[0], _ptr(out), _ptr(workspace), workspace.numel(),
                                         wait_ms, _stream(stream)), "sp_test_expired_wait")

    def w8a8_workspace_size(self, m: int) -> int:
        b = ctypes.c_size_t()
        _check(_lib.sp_w8a8_workspace_size(self._h, m, ctypes.byref(b)), "sp_w8a8_workspace_size")
        return int(b.value)

    def linear_w8a8(self, qx: torch.Tensor, sx: torch.Tensor, out: torch.Tensor | None = None,
                    workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """sp_linear_w8a8: y = sx[m] * sw[n] * (qx . (qw o Mask)^T) for an INT8 matrix, with
        qx [m, K] int8 and sx [m] fp32 per-token scales on this matrix's device."""
        assert qx.dtype == torch.int8 and qx.dim() == 2 and qx.shape[1] == self.k and qx.is_contiguous()
        assert sx.dtype == torch.float32 and sx.shape == (qx.shape[0],) and sx.is_contiguous()
        m = qx.shape[0]
        if out is None:
            out = torch.empty((m, self.n), dtype=torch.bfloat16, device=qx.device)
        if workspace is None:
            workspace = workspace_for(self.w8a8_workspace_size(m), qx.device)
        _check(_lib.sp_linear_w8a8(self._h, _ptr(qx), _ptr(sx), m, _ptr(out), _ptr(workspace), workspace.numel(),
                                   _stream(stream, self.device)), "sp_linear_w8a8")
        return out

    def masked_update(self, grad: torch.Tensor, lr: float, stream=None) -> "SparseMatrix":
        """sp_masked_update: w <- bf16(fma(-lr, grad, w)) on every kept weight, in place on
        the compressed values (Algorithm 1's masked step); grad [N, K] float32 on this
        matrix's device."""
        assert grad.dtype == torch.float32 and grad.shape == (self.n, self.k) and grad.is_contiguous()
        _check(_lib.sp_masked_update(self._h, _ptr(grad), float(lr), _stream(stream, self.device)), "sp_masked_update")
        return self

    def decompress(self, stream=None) -> torch.Tensor:
        dt = torch.int8 if self.dtype == "int8" else torch.bfloat16
        out = torch.empty((self.n, self.k), dtype=dt, device=torch.device("cuda", int(self.info.device)))
        _check(_lib.sp_decompress(self._h, _ptr(out), _stream(stream)), "sp_decompress")
        return out

    def copy_out(self) -> tuple[np.ndarray, np.ndarray]:
        buf = np.zeros(max(int(self.info.bytes), 1), dtype=np.uint8)
        off = np.zeros(int(self.info.tiles * self.info.row_blocks + 1), dtype=np.uint64)
        _check(_lib.sp_copy_out(self._h, buf.ctypes.data_as(ctypes.c_void_p), buf.size,
                                off.ctypes.data_as(ctypes.c_void_p), off.size), "sp_copy_out")
        return buf[:int(self.info.bytes)], off

    def clone(self, stream=None) -> "SparseMatrix":
        h = ctypes.c_void_p()
        _check(_lib.sp_clone(self._h, _ALLOC, _FREE, None, _stream(stream), ctypes.byref(h)), "sp_clone")
        return SparseMatrix(h)

    def free(self):
        if self._h:
            torch.cuda.synchronize()
            _check(_lib.sp_free(self._h), "sp_free")
            self._h = None

    def __del__(self):
        try:
            if self._h:
                _lib.sp_free(self._h)
                self._h = None
        except Exception:
            pass


def compress(w: torch.Tensor, mask: torch.Tensor, scale: torch.Tensor | None = None, stream=None) -> SparseMatrix:
    """Compress W o mask.  w: [N, K] bf16 (or int8 with scale [N] fp32); mask: [N, K] uint8/bool."""
    assert w.is_cuda and w.dim() == 2 and w.is_contiguous()
    if mask.dtype == torch.bool:
        mask = mask.to(torch.uint8)
    assert mask.dtype == torch.uint8 and mask.shape == w.shape and mask.is_contiguous()
    if w.dtype == torch.int8:
        assert scale is not None and scale.dtype == torch.float32 and scale.numel() == w.shape[0]
        dt = SP_INT8
    else:
        assert w.dtype in (torch.bfloat16, torch.int16, torch.uint16) and scale is None
        dt = SP_BF16
    h = ctypes.c_void_p()
    _check(_lib.sp_compress(_ptr(w), _ptr(mask), w.shape[0], w.shape[1], dt, _ptr(scale), _ALLOC, _FREE, None,
                            _stream(stream), ctypes.byref(h)), "sp_compress")
    return SparseMatrix(h)


_ws_cache: dict = {}


def workspace_for(nbytes: int, device) -> torch.Tensor:
    """A zero-filled workspace of at least nbytes on `device`, shared by calls on one stream."""
    dev = torch.device(device)
    key = dev.index if dev.index is not None else torch.cuda.current_device()
    ws = _ws_cache.get(key)
    if ws is None or ws.numel() < max(nbytes, 1):
        ws = torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=torch.device("cuda", key))
        _ws_cache[key] = ws
    return ws


def copy_columns(out: torch.Tensor, inp: torch.Tensor, col0: int, stream=None) -> torch.Tensor:
    """out[m, :] = inp[m, col0 : col0 + out.shape[1]] (bf16, in a libsp kernel)."""
    M, n = out.shape
    _check(_lib.sp_copy_columns(_ptr(out), _ptr(inp), M, inp.shape[1], col0, n, _stream(stream, out.device.index)),
           "sp_copy_columns")
    return out


def residual_add(h: torch.Tensor, a: torch.Tensor, r: torch.Tensor, stream=None) -> torch.Tensor:
    """h = bf16(h + a + r) in place, r broadcast over rows."""
    M, N = h.shape
    _check(_lib.sp_residual_add(_ptr(h), _ptr(a), _ptr(r), M, N, _stream(stream, h.device.index)), "sp_residual_add")
    return h


def mul_pairs(out: torch.Tensor, g: torch.Tensor, stream=None) -> torch.Tensor:
    """out = bf16(g[:, 0::2] * g[:, 1::2]) with F = out.shape[1] (interleaved gate/up rows)."""
    M, F = out.shape
    _check(_lib.sp_mul_pairs(_ptr(out), _ptr(g), M, F, _stream(stream, out.device.index)), "sp_mul_pairs")
    return out


def mul_halves(out: torch.Tensor, g: torch.Tensor, stream=None) -> torch.Tensor:
    """out = bf16(g[:, :F] * g[:, F:]) with F = out.shape[1]."""
    M, F = out.shape
    _check(_lib.sp_mul_halves(_ptr(out), _ptr(g), M, F, _stream(stream, out.device.index)), "sp_mul_halves")
    return out


class Chain:
    """A fixed chain of sparse linears (sp_chain_run): op k reads its x only once op k-1 is
    complete.  Each op is (matrix, x view, y view, epilogue, r); x and y are 2-D bf16 views
    with unit column stride (row stride = their stride(0)).  The ctypes op array is built
    once; run() is one library call per group of up to 160 linears."""

    def __init__(self, ops, m: int):
        self.m = m
        self._keep = []
        arr = (SpChainOp * max(len(ops), 1))()
        for i, (mat, x, y, epi, r) in enumerate(ops):
            assert x.dtype == torch.bfloat16 and y.dtype == torch.bfloat16 and x.stride(1) == 1 and y.stride(1) == 1
            assert x.shape[0] >= m and y.shape[0] >= m and x.shape[1] == mat.k
            assert y.shape[1] == (mat.n // 2 if epi == "pair_product" else mat.n)
            arr[i] = SpChainOp(mat.handle, x.data_ptr(), x.stride(0), y.data_ptr(), y.stride(0),
                               0 if r is None else r.data_ptr(), EPILOGUES[epi], 0)
            self._keep.append((mat, x, y, r))
        self._ops = arr
        self.n_ops = len(ops)
        b = ctypes.c_size_t()
        _check(_lib.sp_chain_workspace_size(m, ctypes.byref(b)), "sp_chain_workspace_size")
        dev = torch.device("cuda", torch.cuda.current_device())
        self.workspace = torch.zeros(max(int(b.value), 256), dtype=torch.uint8, device=dev)

    def run(self, stream=None):
        _check(_lib.sp_chain_run(self._ops, self.n_ops, self.m, _ptr(self.workspace), self.workspace.numel(),
                                 _stream(stream, self.workspace.device.index)), "sp_chain_run")


def check(stream=None):
    """Synchronise the stream and raise if a kernel's bounded wait expired."""
    _check(_lib.sp_check(_stream(stream)), "sp_check")


def status_string(code: int) -> str:
    return _lib.sp_status_string(code).decode()
