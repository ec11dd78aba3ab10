"""The oracle's pins must be sharp: plant one plausible mistake at a time in a copy of
sp_oracle.c (on the CPU), rebuild it, and check that at least one pin fails."""
import os
import subprocess

import pytest

import oracle as oracle_mod
from tests import test_oracle as pins

SRC = os.path.join(os.path.dirname(oracle_mod.__file__), "sp_oracle.c")

# Every mutant keeps the oracle's memory accesses inside its buffers (a mistake that
# corrupts memory would end the test process rather than fail a pin).
MUTANTS = {
    "sum_sign": ("acc += or_bf16_to_double(x[m * K + k]) * or_bf16_to_double(W[n * K + k]);",
                 "acc -= or_bf16_to_double(x[m * K + k]) * or_bf16_to_double(W[n * K + k]);"),
    "transposed_x": ("acc += or_bf16_to_double(x[m * K + k]) * or_bf16_to_double(W[n * K + k]);",
                     "acc += or_bf16_to_double(x[k * M + m]) * or_bf16_to_double(W[n * K + k]);"),
    "dropped_first_term": ("for (int64_t k = 0; k < K; ++k)\n        if (mask[n * K + k]) acc += or_bf16_to_double(x[m * K + k]) * or_bf16_to_double(W",
                           "for (int64_t k = 1; k < K; ++k)\n        if (mask[n * K + k]) acc += or_bf16_to_double(x[m * K + k]) * or_bf16_to_double(W"),
    "mask_msb_first": ("if (k < K && mask[n * K + k]) m |= (uint64_t)1 << j;",
                       "if (k < K && mask[n * K + k]) m |= (uint64_t)1 << (63 - j);"),
    "pad_to_8": ("#define OR_ALIGN 16", "#define OR_ALIGN 8"),
    "int8_scale_dropped": ("acc += or_bf16_to_double(x[m * K + k]) * ((double)q[n * K + k] * sn);",
                           "acc += or_bf16_to_double(x[m * K + k]) * ((double)q[n * K + k]);"),
    "block_mask_msb_first": ("m |= (uint64_t)1 << i;", "m |= (uint64_t)1 << (n - 1 - i);"),
    "residual_r_dropped": (" + or_bf16_to_double(a[m * N + j]) + or_bf16_to_double(r[j]);",
                           " + or_bf16_to_double(a[m * N + j]);"),
    "halves_row_stride": ("or_bf16_to_double(g[m * 2 * F + j]) * or_bf16_to_double(g[m * 2 * F + F + j])",
                          "or_bf16_to_double(g[m * F + j]) * or_bf16_to_double(g[m * F + F + j])"),
    "w8a8_token_scale": ("y[m * N + n] = ((double)sx[m] * (double)sw[n]) * (double)acc;",
                         "y[m * N + n] = ((double)sx[0] * (double)sw[n]) * (double)acc;"),
    "w8a8_mask_dropped": ("if (mask[n * K + k]) acc += (int64_t)qx[m * K + k] * (int64_t)qw[n * K + k];",
                          "acc += (int64_t)qx[m * K + k] * (int64_t)qw[n * K + k];"),
    "w8a8_unsigned": ("if (mask[n * K + k]) acc += (int64_t)qx[m * K + k] * (int64_t)qw[n * K + k];",
                      "if (mask[n * K + k]) acc += (int64_t)(uint8_t)qx[m * K + k] * (int64_t)qw[n * K + k];"),
    "update_sign": ("h = or_float_to_bf16_rne(fmaf(-lr, grad[n * K + k], w));",
                    "h = or_float_to_bf16_rne(fmaf(lr, grad[n * K + k], w));"),
    "update_truncates": ("u += 0x7FFFu + ((u >> 16) & 1u);", "u += 0u;"),
    "update_grad_index": ("h = or_float_to_bf16_rne(fmaf(-lr, grad[n * K + k], w));",
                          "h = or_float_to_bf16_rne(fmaf(-lr, grad[n * K + (k ^ 1)], w));"),
    "bf16_shift": ("uint32_t u = (uint32_t)h << 16;", "uint32_t u = (uint32_t)h << 15;"),
    "decompress_value_not_advanced": ("memcpy(Wb + (n * K + k) * esize, vals + v * esize, (size_t)esize);\n          ++v;",
                                      "memcpy(Wb + (n * K + k) * esize, vals + v * esize, (size_t)esize);"),
    "decompress_chunks_transposed": ("const uint8_t* chunk = buf + off[rb * T + t];\n      const uint8_t* vals = chunk + OR_MASK_BYTES;\n      int64_t v = 0;\n      for (int r = 0; r < OR_CHUNK_ROWS; ++r) {\n        int64_t n = rb * OR_CHUNK_ROWS + r;\n        uint64_t m = or_read_u64le",
                                     "const uint8_t* chunk = buf + off[t * RB + rb];\n      const uint8_t* vals = chunk + OR_MASK_BYTES;\n      int64_t v = 0;\n      for (int r = 0; r < OR_CHUNK_ROWS; ++r) {\n        int64_t n = rb * OR_CHUNK_ROWS + r;\n        uint64_t m = or_read_u64le"),
    "from_format_byte_swap": ("uint16_t h = (uint16_t)(vals[2 * v] | (vals[2 * v + 1] << 8));",
                              "uint16_t h = (uint16_t)(vals[2 * v + 1] | (vals[2 * v] << 8));"),
    "from_format_neighbour_mask": ("uint64_t msk = or_read_u64le(chunk + r * 8);",
                                   "uint64_t msk = or_read_u64le(chunk + (r ^ 1) * 8);"),
    "from_format_int8_unscaled": ("w = (double)(int8_t)vals[v] * (double)scale[n];", "w = (double)(int8_t)vals[v];"),
    "from_format_int8_unsigned": ("w = (double)(int8_t)vals[v] * (double)scale[n];",
                                  "w = (double)vals[v] * (double)scale[n];"),
    "residual_h_dropped": ("out[m * N + j] = or_bf16_to_double(h[m * N + j]) + or_bf16_to_double(a[m * N + j])",
                           "out[m * N + j] = or_bf16_to_double(a[m * N + j]) + or_bf16_to_double(a[m * N + j])"),
    "tile_width_off_by_one": ("for (int j = 0; j < OR_TILE_K; ++j) {\n          if (!((m >> j) & 1u)) continue;\n          int64_t k = t * OR_TILE_K + j;\n          memcpy(vals",
                              "for (int j = 1; j < OR_TILE_K; ++j) {\n          if (!((m >> j) & 1u)) continue;\n          int64_t k = t * OR_TILE_K + j;\n          memcpy(vals"),
}


def _pin_suite(o):
    """Run a fixed selection of pins against whatever library `o` is bound to; return
    the names of those that failed."""
    checks = {
        "paper_example": lambda: pins.test_paper_example_register_layout_and_encoding(o),
        "format_bytes": lambda: pins.test_format_hand_derived_bytes(o),
        "format_linear": lambda: pins.test_format_hand_derived_linear(o),
        "roundtrip": lambda: pins.test_roundtrip_bit_exact(o, 300, 200, 70, False),
        "roundtrip_int8": lambda: pins.test_roundtrip_bit_exact(o, 130, 72, 50, True),
        "layout": lambda: pins.test_layout_invariants(o, 257, 136),
        "integer_exact": lambda: pins.test_linear_integer_valued_exact(o, 40, 136, 3),
        "library_matmul": lambda: pins.test_linear_matches_float64_library_matmul(o, 70),
        "one_hot": lambda: pins.test_linear_one_hot_selects_a_column(o),
        "from_format_def": lambda: pins.test_linear_from_format_bitwise_equals_definition(o),
        "int8_exact": lambda: pins.test_int8_oracle_integer_exact_and_scale(o),
        "glue": lambda: pins.test_glue_hand_derived_values(o),
        "w8a8_int": lambda: pins.test_w8a8_integer_sum_equals_int64_matmul(o),
        "w8a8_scales": lambda: pins.test_w8a8_scales_by_token_and_by_row(o),
        "update_rounding": lambda: pins.test_masked_update_hand_derived_rounding(o),
        "update_dense": lambda: pins.test_masked_update_equals_dense_step_then_compress(o),
    }
    failed = []
    for name, fn in checks.items():
        try:
            fn()
        except (AssertionError, ValueError):
            failed.append(name)
    return failed


def test_unmutated_oracle_passes_the_suite(oracle):
    assert _pin_suite(oracle) == []


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_each_planted_mistake_is_caught(oracle, tmp_path, name):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) >= 1, f"mutation anchor for {name} not found"
    mutated = src.replace(old, new, 1)
    path_c = tmp_path / "mut.c"
    path_c.write_text(mutated)
    so = tmp_path / "libmut.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", str(path_c), "-o", str(so), "-lm"])
    oracle_mod.use_library(str(so))
    try:
        failed = _pin_suite(oracle_mod)
    finally:
        oracle_mod.use_library(None)
    assert failed, f"mutant {name} survived every pin"
