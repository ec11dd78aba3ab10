"""Host logic of the linear stack, on the CPU: the gate/up row interleave that lets the
gate * up product be an epilogue over row pairs (2j, 2j + 1) of one linear."""
import numpy as np

from paper_2405_03594_gb300 import synth
from paper_2405_03594_gb300.stack import interleave_rows


def test_interleave_is_the_pairing_permutation():
    F, K = 5, 3
    a = np.arange(2 * F * K).reshape(2 * F, K)
    b = interleave_rows(a, F)
    for j in range(F):
        assert np.array_equal(b[2 * j], a[j]) and np.array_equal(b[2 * j + 1], a[F + j])
    assert sorted(map(tuple, b)) == sorted(map(tuple, a))
    s = np.arange(2 * F, dtype=np.float32)  # per-row scales follow their rows
    assert list(interleave_rows(s, F)) == [0, 5, 1, 6, 2, 7, 3, 8, 4, 9]


def test_pair_products_of_interleaved_rows_are_gate_times_up(oracle):
    """y over the interleaved weight, multiplied in row pairs, equals gate * up of the
    [gate, up] layout: the product the glue sp_mul_halves takes on the plain layout."""
    F, K, M = 96, 136, 3
    g = np.random.default_rng(4)
    W = synth.weight(2 * F, K, g)
    mask = synth.magnitude_mask(W, 70)
    x = synth.activations(M, K, g)
    y = oracle.linear_bf16(x, interleave_rows(W, F), interleave_rows(mask, F))
    plain = oracle.linear_bf16(x, W, mask)
    assert np.array_equal(y[:, 0::2], plain[:, :F]) and np.array_equal(y[:, 1::2], plain[:, F:])
    pairs = y[:, 0::2] * y[:, 1::2]
    assert np.array_equal(pairs, plain[:, :F] * plain[:, F:])


def test_interleaved_int8_rows_keep_their_scales(oracle):
    F, K, M = 40, 72, 2
    g = np.random.default_rng(6)
    W = synth.weight(2 * F, K, g)
    mask = synth.magnitude_mask(W, 50)
    q, s = synth.quantize_int8(W, mask)
    x = synth.activations(M, K, g)
    y = oracle.linear_int8(x, interleave_rows(q, F), interleave_rows(mask, F), interleave_rows(s, F))
    plain = oracle.linear_int8(x, q, mask, s)
    assert np.array_equal(y[:, 0::2], plain[:, :F]) and np.array_equal(y[:, 1::2], plain[:, F:])
