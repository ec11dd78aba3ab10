"""The ctypes binding mirrors the C declarations of include/sp.h and include/sp_stack.h:
struct sizes, field offsets and enum values, checked against a C program compiled from the
headers (gcc, no GPU)."""
import ctypes
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

C_SRC = r"""
#include <stddef.h>
#include <stdio.h>
#include "sp_stack.h"
int main(void) {
  printf("sp_chain_op %zu\n", sizeof(sp_chain_op));
  printf("sp_chain_op.w %zu\n", offsetof(sp_chain_op, w));
  printf("sp_chain_op.x %zu\n", offsetof(sp_chain_op, x));
  printf("sp_chain_op.ldx %zu\n", offsetof(sp_chain_op, ldx));
  printf("sp_chain_op.y %zu\n", offsetof(sp_chain_op, y));
  printf("sp_chain_op.ldy %zu\n", offsetof(sp_chain_op, ldy));
  printf("sp_chain_op.r %zu\n", offsetof(sp_chain_op, r));
  printf("sp_chain_op.epilogue %zu\n", offsetof(sp_chain_op, epilogue));
  printf("sp_chain_op.reserved %zu\n", offsetof(sp_chain_op, reserved));
  printf("sp_info_t %zu\n", sizeof(sp_info_t));
  printf("sp_info_t.n %zu\n", offsetof(sp_info_t, n));
  printf("sp_info_t.k %zu\n", offsetof(sp_info_t, k));
  printf("sp_info_t.tiles %zu\n", offsetof(sp_info_t, tiles));
  printf("sp_info_t.row_blocks %zu\n", offsetof(sp_info_t, row_blocks));
  printf("sp_info_t.dtype %zu\n", offsetof(sp_info_t, dtype));
  printf("sp_info_t.device %zu\n", offsetof(sp_info_t, device));
  printf("sp_info_t.nnz %zu\n", offsetof(sp_info_t, nnz));
  printf("sp_info_t.bytes %zu\n", offsetof(sp_info_t, bytes));
  printf("sp_info_t.max_chunk_bytes %zu\n", offsetof(sp_info_t, max_chunk_bytes));
  printf("sp_info_t.scale_bytes %zu\n", offsetof(sp_info_t, scale_bytes));
  printf("SP_EPI_STORE %d\nSP_EPI_RESIDUAL %d\nSP_EPI_PAIR_PRODUCT %d\n", SP_EPI_STORE, SP_EPI_RESIDUAL,
         SP_EPI_PAIR_PRODUCT);
  printf("SP_BF16 %d\nSP_INT8 %d\n", SP_BF16, SP_INT8);
  printf("SP_PATH_AUTO %d\nSP_PATH_CUDA_CORE %d\nSP_PATH_TENSOR_CORE %d\n", SP_PATH_AUTO, SP_PATH_CUDA_CORE,
         SP_PATH_TENSOR_CORE);
  return 0;
}
"""


@pytest.fixture(scope="module")
def c_layout(tmp_path_factory):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not found")
    d = tmp_path_factory.mktemp("abi")
    src, exe = d / "layout.c", d / "layout"
    src.write_text(C_SRC)
    subprocess.check_call([gcc, "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)])
    out = subprocess.check_output([str(exe)], text=True)
    return {k: int(v) for k, v in (line.split() for line in out.strip().splitlines())}


def _binding_types():
    """The binding's ctypes declarations, without loading libsp.so (they are module-level
    classes; the module itself needs the built library)."""
    import ast

    src = open(os.path.join(ROOT, "paper_2405_03594_gb300", "sp.py")).read()
    tree = ast.parse(src)
    ns = {"ctypes": ctypes}
    for node in tree.body:
        if isinstance(node, ast.ClassDef) and node.name in ("SpInfo", "SpChainOp"):
            exec(compile(ast.Module(body=[node], type_ignores=[]), "sp.py", "exec"), ns)
        if isinstance(node, ast.Assign) and any(getattr(t, "id", "") in ("EPILOGUES", "PATHS") for t in node.targets):
            exec(compile(ast.Module(body=[node], type_ignores=[]), "sp.py", "exec"), ns)
        if isinstance(node, ast.Assign) and any(isinstance(t, ast.Tuple) for t in node.targets):
            names = [e.id for t in node.targets if isinstance(t, ast.Tuple) for e in t.elts]
            if "SP_BF16" in names:
                exec(compile(ast.Module(body=[node], type_ignores=[]), "sp.py", "exec"), ns)
    return ns


def test_chain_op_layout(c_layout):
    ns = _binding_types()
    T = ns["SpChainOp"]
    assert ctypes.sizeof(T) == c_layout["sp_chain_op"]
    for f in ("w", "x", "ldx", "y", "ldy", "r", "epilogue", "reserved"):
        assert getattr(T, f).offset == c_layout[f"sp_chain_op.{f}"], f


def test_info_layout(c_layout):
    ns = _binding_types()
    T = ns["SpInfo"]
    assert ctypes.sizeof(T) == c_layout["sp_info_t"]
    for f in ("n", "k", "tiles", "row_blocks", "dtype", "device", "nnz", "bytes", "max_chunk_bytes", "scale_bytes"):
        assert getattr(T, f).offset == c_layout[f"sp_info_t.{f}"], f


def test_enum_values(c_layout):
    ns = _binding_types()
    assert ns["EPILOGUES"] == {"store": c_layout["SP_EPI_STORE"], "residual": c_layout["SP_EPI_RESIDUAL"],
                               "pair_product": c_layout["SP_EPI_PAIR_PRODUCT"]}
    assert (ns["SP_BF16"], ns["SP_INT8"]) == (c_layout["SP_BF16"], c_layout["SP_INT8"])
    assert ns["PATHS"] == {"auto": c_layout["SP_PATH_AUTO"], "cuda_core": c_layout["SP_PATH_CUDA_CORE"],
                           "tensor_core": c_layout["SP_PATH_TENSOR_CORE"]}
