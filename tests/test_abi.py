"""The C ABI library loads and exports every function include/sp.h declares; argument
checks that return before touching the GPU behave as documented.  CPU only: no call
here launches a kernel."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", h) for h in sorted(os.listdir(os.path.join(ROOT, "include")))
           if h.endswith(".h")]


@pytest.fixture(scope="module")
def lib():
    from paper_2405_03594_gb300 import build

    path = build.build()
    from paper_2405_03594_gb300 import sp

    assert os.path.samefile(sp.LIB_PATH, path)
    return sp._lib


def declared_functions():
    names = set()
    for hdr in HEADERS:
        src = re.sub(r"/\*.*?\*/", "", open(hdr).read(), flags=re.S)
        names |= set(re.findall(r"^\s*(?:sp_status|const char\s*\*)\s+(sp_\w+)\s*\(", src, flags=re.M))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ["sp_compress", "sp_decompress", "sp_linear", "sp_free", "sp_workspace_size", "sp_check",
              "sp_residual_add", "sp_mul_halves", "sp_copy_columns"]:
        assert n in names


def test_glue_argument_checks(lib):
    P = ctypes.c_void_p
    f = P(1 << 20)
    assert lib.sp_residual_add(None, f, f, 2, 8, None) == 1
    assert lib.sp_residual_add(f, f, f, 2, 12, None) == 2
    assert lib.sp_residual_add(P((1 << 20) + 4), f, f, 2, 8, None) == 3
    assert lib.sp_mul_halves(f, f, 2, 0, None) == 0  # empty: nothing to launch
    assert lib.sp_copy_columns(f, f, 2, 16, 8, 16, None) == 1  # in_stride < col0 + ncols


def test_every_declared_symbol_is_exported(lib):
    from paper_2405_03594_gb300 import sp

    names = declared_functions()
    assert sorted(sp.EXPORTS) == names
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(lib):
    from paper_2405_03594_gb300 import sp

    for code in range(9):
        assert sp.status_string(code) and sp.status_string(code) != "unknown status"
    assert sp.status_string(99) == "unknown status"


def _compress(lib, w, m, n, k, dtype=0, scale=None, out=True):
    from paper_2405_03594_gb300 import sp

    h = ctypes.c_void_p(123)
    rc = lib.sp_compress(ctypes.c_void_p(w), ctypes.c_void_p(m), n, k, dtype, ctypes.c_void_p(scale),
                         sp.ALLOC_FN(), sp.FREE_FN(), None, None, ctypes.byref(h) if out else None)
    return rc, h


def test_compress_argument_checks(lib):
    fake = 1 << 20  # never dereferenced: every case below fails before any CUDA call
    assert _compress(lib, fake, fake, 4, 8, out=False)[0] == 1
    rc, h = _compress(lib, 0, fake, 4, 8)
    assert rc == 1 and h.value is None  # *out cleared on error
    assert _compress(lib, fake, 0, 4, 8)[0] == 1
    assert _compress(lib, fake, fake, 0, 8)[0] == 1
    assert _compress(lib, fake, fake, 4, -8)[0] == 1
    assert _compress(lib, fake, fake, 4, 8, dtype=7)[0] == 1
    assert _compress(lib, fake, fake, 4, 8, dtype=1)[0] == 1  # INT8 needs scales
    assert _compress(lib, fake, fake, 4, 8, dtype=0, scale=fake)[0] == 1  # bf16 takes none
    assert _compress(lib, fake, fake, 4, 100)[0] == 2  # K % 8 != 0: unsupported
    assert _compress(lib, fake + 2, fake, 4, 8)[0] == 3
    assert _compress(lib, fake, fake + 8, 4, 8)[0] == 3


def test_handle_checks(lib):
    P = ctypes.c_void_p
    assert lib.sp_free(None) == 0
    assert lib.sp_info(None, None) == 7
    assert lib.sp_decompress(None, P(1 << 20), None) == 7
    sz = ctypes.c_size_t()
    assert lib.sp_workspace_size(None, 4, ctypes.byref(sz)) == 7
    assert lib.sp_linear(None, P(1 << 20), 1, P(1 << 20), None, 0, None) == 7
    assert lib.sp_linear_ex(None, P(1 << 20), 1, P(1 << 20), None, 0, 0, None) == 7
    n = ctypes.c_int64()
    assert lib.sp_launch_count(None, 4, 0, ctypes.byref(n), None) == 7
    assert lib.sp_masked_update(None, P(1 << 20), ctypes.c_float(0.1), None) == 7
    assert lib.sp_linear_w8a8(None, P(1 << 20), P(1 << 20), 1, P(1 << 20), None, 0, None) == 7
    assert lib.sp_w8a8_workspace_size(None, 4, ctypes.byref(sz)) == 7
    assert lib.sp_linear_epi(None, P(1 << 20), 1, P(1 << 20), 0, None, None, 0, None) == 7
    assert lib.sp_mul_pairs(None, P(1 << 20), 1, 8, None) == 1  # no output
    assert lib.sp_mul_pairs(P(1 << 20), P(1 << 20), 1, 12, None) == 2  # F % 8 != 0
    # a pointer that is not a handle is rejected by its magic word
    junk = (ctypes.c_uint32 * 64)()
    assert lib.sp_info(ctypes.cast(junk, P), None) == 7
    assert lib.sp_free(ctypes.cast(junk, P)) == 7


def test_no_gpu_means_cuda_error_not_a_fallback(lib):
    import torch

    if torch.cuda.is_available():
        pytest.skip("this check is for hosts without a GPU")
    assert lib.sp_check(None) == 4
