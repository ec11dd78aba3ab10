"""Pins for the CPU oracle: each test fixes the oracle to something other than itself
(the paper's worked example, hand-derived bytes, closed forms, integer arithmetic,
a library matmul, invariants).  CPU only."""
import os

import numpy as np
import pytest

from paper_2405_03594_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    d = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            k, v = line.split(":", 1)
            d[k.strip()] = v.split()
    return d


# ---------------------------------------------------------------- Sec. 2.4.1 example


def test_paper_example_register_layout_and_encoding(oracle):
    g = _read_golden("paper_bitmask_example.txt")
    rows = [g["row0"], g["row1"]]
    # Our reading of the VNNI layout: columns in order, the two rows interleaved.
    derived = [rows[i % 2][i // 2] for i in range(16)]
    assert derived == g["register_layout"]
    # Give every symbol a distinct nonzero int16 and encode the block in register order.
    sym = {s: 100 + i for i, s in enumerate(sorted({t for t in derived if t != "0"}))}
    elems = [0 if t == "0" else sym[t] for t in derived]
    values, mask = oracle.block_encode(elems)
    assert values == [sym[s] for s in g["values"]]
    assert bin(mask).count("1") == 9 == len(g["values"])
    printed = g["bitmask_printed"][0]
    assert printed.startswith("0b")
    digits = printed[2:]
    # Reading the printed digits with element 0 leftmost gives our LSB-first mask ...
    assert mask == sum(1 << i for i, ch in enumerate(digits) if ch == "1")
    assert mask == 0xE94E
    # ... while the literal read as an ordinary binary number is a different integer.
    assert int(printed, 2) == 0x7297 != mask


# ---------------------------------------------------------------- format bytes


def _golden_2x8():
    g = _read_golden("format_2x8.txt")
    N, K = int(g["N"][0]), int(g["K"][0])
    W = np.array([[int(h, 16) for h in g["W_row0_bf16"]], [int(h, 16) for h in g["W_row1_bf16"]]], dtype=np.uint16)
    mask = np.array([[int(v) for v in g["mask_row0"]], [int(v) for v in g["mask_row1"]]], dtype=np.uint8)
    return g, N, K, W, mask


def test_format_hand_derived_bytes(oracle):
    g, N, K, W, mask = _golden_2x8()
    buf, off = oracle.compress(W, mask)
    total = int(g["expect_total_bytes"][0])
    assert buf.size == total and list(off) == [0, total]
    masks = buf[:1024].view(np.uint64)
    exp_m = [int(v, 16) for v in g["expect_mask_u64"]]
    assert list(masks[:2]) == exp_m and not masks[2:].any()
    vb = [int(v, 16) for v in g["expect_value_bytes"]]
    assert list(buf[1024:1024 + len(vb)]) == vb
    assert not buf[1024 + len(vb):].any()


def test_format_hand_derived_linear(oracle):
    g, N, K, W, mask = _golden_2x8()
    x = synth.bf16_from_f32(np.array([[float(v) for v in g["x_row0"]], [float(v) for v in g["x_row1"]]], np.float32))
    y = oracle.linear_bf16(x, W, mask)
    exp = np.array([[float(v) for v in g["expect_y_row0"]], [float(v) for v in g["expect_y_row1"]]])
    assert np.array_equal(y, exp)
    buf, off = oracle.compress(W, mask)
    assert np.array_equal(oracle.linear_from_format(buf, off, N, K, 2, x), exp)


# ---------------------------------------------------------------- round trip and invariants

SHAPES = [(1, 8), (2, 64), (130, 72), (300, 200), (257, 136), (128, 1024)]


def _rand_case(N, K, pct, seed, int8=False):
    g = np.random.default_rng(seed)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    if int8:
        q, s = synth.quantize_int8(W, mask)
        return q, mask, s
    return W, mask, None


@pytest.mark.parametrize("N,K", SHAPES)
@pytest.mark.parametrize("pct", [0, 50, 70, 100])
@pytest.mark.parametrize("int8", [False, True])
def test_roundtrip_bit_exact(oracle, N, K, pct, int8):
    W, mask, _ = _rand_case(N, K, pct, seed=N * 7 + K + pct, int8=int8)
    buf, off = oracle.compress(W, mask)
    back = oracle.decompress(buf, off, N, K, W.dtype)
    expect = np.where(mask != 0, W, np.zeros_like(W))
    assert np.array_equal(back.view(np.uint8), expect.view(np.uint8))


@pytest.mark.parametrize("N,K", SHAPES)
def test_layout_invariants(oracle, N, K):
    W, mask, _ = _rand_case(N, K, 60, seed=3)
    buf, off = oracle.compress(W, mask)
    T, RB = oracle.geometry(N, K)
    assert off.size == RB * T + 1 and off[0] == 0 and off[-1] == buf.size
    sizes = np.diff(off.astype(np.int64))
    assert (sizes % 16 == 0).all() and (sizes >= 1024 + 0).all()
    total_bits = 0
    for c in range(RB * T):
        rb, t = divmod(c, T)
        chunk = buf[int(off[c]):int(off[c + 1])]
        m = chunk[:1024].view(np.uint64)
        bits = sum(bin(int(v)).count("1") for v in m)
        total_bits += bits
        # chunk size is exactly masks + packed values, padded to 16
        assert sizes[c] == (1024 + 2 * bits + 15) // 16 * 16
        assert not chunk[1024 + 2 * bits:].any()
        # rows past N and columns past K carry no bits
        for r in range(128):
            n = rb * 128 + r
            valid = min(64, K - 64 * t)
            if n >= N:
                assert m[r] == 0
            elif valid < 64:
                assert int(m[r]) >> valid == 0
    assert total_bits == int(mask.sum())


def test_masked_in_zero_kept_and_negative_zero_preserved(oracle):
    N, K = 3, 16
    W = np.zeros((N, K), dtype=np.uint16)
    W[0, 3] = 0x8000  # -0.0, kept
    W[1, 5] = 0x3F80  # 1.0, masked out: dropped
    W[2, 7] = 0x0000  # +0.0, kept: stored as a value
    mask = np.zeros((N, K), dtype=np.uint8)
    mask[0, 3] = 1
    mask[2, 7] = 1
    buf, off = oracle.compress(W, mask)
    vals = buf[1024:1028].view(np.uint16)
    assert list(vals) == [0x8000, 0x0000]
    back = oracle.decompress(buf, off, N, K, np.uint16)
    assert back[0, 3] == 0x8000 and back[1, 5] == 0 and back[2, 7] == 0


# ---------------------------------------------------------------- the product


@pytest.mark.parametrize("N,K", [(5, 8), (40, 136), (129, 200), (64, 64)])
@pytest.mark.parametrize("M", [1, 3, 8])
def test_linear_integer_valued_exact(oracle, N, K, M):
    """Integer-valued inputs: every product and partial sum is an exact small integer,
    so the float64 oracle must equal an int64 matmul of the masked weight exactly."""
    g = np.random.default_rng(N * 1000 + K + M)
    Wi = g.integers(-4, 5, size=(N, K))
    xi = g.integers(-2, 3, size=(M, K))
    mask = (g.random((N, K)) < 0.4).astype(np.uint8)
    W = synth.bf16_from_f32(Wi.astype(np.float32))
    x = synth.bf16_from_f32(xi.astype(np.float32))
    y = oracle.linear_bf16(x, W, mask)
    exact = xi @ (Wi * mask).T
    assert np.array_equal(y, exact.astype(np.float64))
    buf, off = oracle.compress(W, mask)
    assert np.array_equal(oracle.linear_from_format(buf, off, N, K, 2, x), y)


@pytest.mark.parametrize("pct", [0, 50, 70, 80])
def test_linear_matches_float64_library_matmul(oracle, pct):
    N, K, M = 200, 264, 5
    g = np.random.default_rng(pct)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    x = synth.activations(M, K, g)
    y = oracle.linear_bf16(x, W, mask)
    Wd = synth.bf16_to_f32(W).astype(np.float64) * mask
    ref = synth.bf16_to_f32(x).astype(np.float64) @ Wd.T
    assert np.allclose(y, ref, rtol=1e-12, atol=1e-14)
    # transposed-operand mistakes would not survive a non-square, non-symmetric case
    assert y.shape == (M, N)


def test_linear_from_format_bitwise_equals_definition(oracle):
    N, K, M = 300, 200, 4
    g = np.random.default_rng(11)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, 70)
    x = synth.activations(M, K, g)
    buf, off = oracle.compress(W, mask)
    assert np.array_equal(oracle.linear_from_format(buf, off, N, K, 2, x), oracle.linear_bf16(x, W, mask))


def test_linear_one_hot_selects_a_column(oracle):
    N, K = 130, 136
    g = np.random.default_rng(5)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, 50)
    ks = [0, 1, 63, 64, 65, 127, 128, 135]
    x = np.zeros((len(ks), K), dtype=np.uint16)
    for i, k in enumerate(ks):
        x[i, k] = 0x3F80
    y = oracle.linear_bf16(x, W, mask)
    Wf = synth.bf16_to_f32(W).astype(np.float64) * mask
    for i, k in enumerate(ks):
        assert np.array_equal(y[i], Wf[:, k])


def test_linear_empty_rows_give_zero(oracle):
    N, K, M = 20, 64, 2
    g = np.random.default_rng(2)
    W = synth.weight(N, K, g)
    mask = np.ones((N, K), dtype=np.uint8)
    mask[[0, 7, 19]] = 0
    x = synth.activations(M, K, g)
    y = oracle.linear_bf16(x, W, mask)
    assert (y[:, [0, 7, 19]] == 0).all() and (y[:, 1] != 0).all()


def test_int8_oracle_integer_exact_and_scale(oracle):
    N, K, M = 70, 136, 3
    g = np.random.default_rng(9)
    q = g.integers(-127, 128, size=(N, K)).astype(np.int8)
    mask = (g.random((N, K)) < 0.3).astype(np.uint8)
    xi = g.integers(-2, 3, size=(M, K))
    x = synth.bf16_from_f32(xi.astype(np.float32))
    ones = np.ones(N, dtype=np.float32)
    y1 = oracle.linear_int8(x, q, mask, ones)
    exact = xi @ (q.astype(np.int64) * mask).T
    assert np.array_equal(y1, exact.astype(np.float64))
    s = (g.random(N).astype(np.float32) + 0.5) / 64
    ys = oracle.linear_int8(x, q, mask, s)
    # integer sums below 2^24 times an fp32 scale are exact in float64
    assert np.array_equal(ys, exact * s.astype(np.float64)[None, :])
    buf, off = oracle.compress(q, mask)
    assert np.array_equal(oracle.linear_from_format(buf, off, N, K, 1, x, s), ys)


# ---------------------------------------------------------------- stack glue

# bf16 bit patterns of exactly representable values (sign, 8-bit exponent, 7-bit mantissa):
# 1.0 = 0x3F80, 1.5 = 0x3FC0, -0.25 = 0xBE80, 2.0 = 0x4000, -3.0 = 0xC040, 10.0 = 0x4120,
# 0.125 = 0x3E00, 0.5 = 0x3F00, 4.0 = 0x4080, -1.0 = 0xBF80.
_BF = {1.0: 0x3F80, 1.5: 0x3FC0, -0.25: 0xBE80, 2.0: 0x4000, -3.0: 0xC040, 10.0: 0x4120,
       0.125: 0x3E00, 0.5: 0x3F00, 4.0: 0x4080, -1.0: 0xBF80}


def _bits(rows):
    return np.array([[_BF[v] for v in row] for row in rows], dtype=np.uint16)


def test_bf16_bit_patterns_are_the_values():
    for v, b in _BF.items():
        assert np.array([b << 16], dtype=np.uint32).view(np.float32)[0] == v


def test_glue_hand_derived_values(oracle):
    """Residual add h + a + r with r broadcast over the rows, and the gate/up product of a
    row laid out as [gate_0 .. gate_{F-1}, up_0 .. up_{F-1}]; expected values by hand."""
    h = _bits([[1.5, -0.25, 2.0], [1.0, -3.0, 10.0]])
    a = _bits([[2.0, 1.0, 0.125], [-0.25, 1.5, -3.0]])
    r = _bits([[10.0, 0.125, -1.0]])[0]
    out = oracle.residual_add(h, a, r)
    assert np.array_equal(out, np.array([[13.5, 0.875, 1.125], [10.75, -1.375, 6.0]]))
    g = _bits([[1.5, -0.25, 2.0, 4.0], [-3.0, 0.5, 10.0, 0.125]])
    out = oracle.mul_halves(g)
    assert np.array_equal(out, np.array([[3.0, -1.0], [-30.0, 0.0625]]))


# ---------------------------------------------------------------- INT8 weights and activations (Sec. 3.4)


def _w8a8_case(M, N, K, seed):
    g = np.random.default_rng(seed)
    qx = g.integers(-127, 128, size=(M, K)).astype(np.int8)
    qw = g.integers(-127, 128, size=(N, K)).astype(np.int8)
    mask = (g.random((N, K)) < 0.3).astype(np.uint8)
    return qx, qw, mask


def test_w8a8_integer_sum_equals_int64_matmul(oracle):
    qx, qw, mask = _w8a8_case(3, 70, 136, 21)
    acc, y = oracle.linear_w8a8(qx, np.ones(3, np.float32), qw, mask, np.ones(70, np.float32))
    exact = qx.astype(np.int64) @ (qw.astype(np.int64) * mask).T
    assert np.array_equal(acc, exact) and np.array_equal(y, exact.astype(np.float64))


def test_w8a8_scales_by_token_and_by_row(oracle):
    """Power-of-two scales keep everything exact: y[m, n] = acc[m, n] * 2^m * 2^-(n % 5)."""
    M, N, K = 4, 37, 72
    qx, qw, mask = _w8a8_case(M, N, K, 22)
    sx = (2.0 ** np.arange(M)).astype(np.float32)
    sw = (2.0 ** -(np.arange(N) % 5)).astype(np.float32)
    acc, y = oracle.linear_w8a8(qx, sx, qw, mask, sw)
    assert np.array_equal(y, acc * (2.0 ** np.arange(M))[:, None] * (2.0 ** -(np.arange(N) % 5))[None, :])


def test_w8a8_matches_int8_weights_with_exact_bf16_activations(oracle):
    """With sx a power of two, x = qx * sx is exact in bf16 (|qx| <= 127), and the INT8-weight
    oracle with bf16 x must give the same float64 result (every partial sum is exact)."""
    M, N, K = 2, 50, 200
    qx, qw, mask = _w8a8_case(M, N, K, 23)
    sx = np.full(M, 2.0 ** -6, np.float32)
    sw = (np.random.default_rng(24).random(N).astype(np.float32) + 0.5) / 64
    _, y = oracle.linear_w8a8(qx, sx, qw, mask, sw)
    x = synth.bf16_from_f32(qx.astype(np.float32) * sx[:, None])
    assert np.array_equal(synth.bf16_to_f32(x), qx.astype(np.float32) * sx[:, None])
    assert np.array_equal(oracle.linear_int8(x, qw, mask, sw), y)


# ---------------------------------------------------------------- masked update (Sec. 2.1, Algorithm 1)


def _one_entry_update(oracle, w_bits, g, lr):
    """Compress a 3 x 72 matrix whose only kept entry is (1, 5) = w_bits, apply the masked
    step with gradient g there (and 1e30 everywhere else), return the updated entry's bits."""
    N, K = 3, 72
    W = np.zeros((N, K), dtype=np.uint16)
    W[1, 5] = w_bits
    mask = np.zeros((N, K), dtype=np.uint8)
    mask[1, 5] = 1
    grad = np.full((N, K), 1e30, dtype=np.float32)
    grad[1, 5] = g
    buf, off = oracle.compress(W, mask)
    out = oracle.masked_update_bf16(buf, off, N, K, grad, lr)
    back = oracle.decompress(out, off, N, K, np.uint16)
    assert not np.delete(back.ravel(), 1 * K + 5).any()
    assert np.array_equal(out[:1024], buf[:1024]) and out.size == buf.size
    return int(back[1, 5])


def test_masked_update_hand_derived_rounding(oracle):
    """w - lr*g rounded once to bf16, nearest-even: 1 + 2^-8 lies halfway between 1.0
    (0x3F80, even) and 1 + 2^-7 (0x3F81); 1 + 3*2^-8 halfway between 0x3F81 and 0x3F82
    (even); 1 + 2^-8 + 2^-20 just above halfway.  The other cases are exact."""
    assert _one_entry_update(oracle, 0x3F80, -2.0 ** -8, 1.0) == 0x3F80
    assert _one_entry_update(oracle, 0x3F80, -3 * 2.0 ** -8, 1.0) == 0x3F82
    assert _one_entry_update(oracle, 0x3F80, -(2.0 ** -8 + 2.0 ** -20), 1.0) == 0x3F81
    assert _one_entry_update(oracle, 0x4000, 4.0, 0.5) == 0x0000      # 2 - 0.5*4 = +0
    assert _one_entry_update(oracle, 0xBFC0, 2.0, 0.25) == 0xC000     # -1.5 - 0.25*2 = -2
    assert _one_entry_update(oracle, 0x3F80, 1.0, -1.0) == 0x4000     # 1 + 1 = 2 (negative step)


def test_masked_update_equals_dense_step_then_compress(oracle):
    """Algorithm 1 written densely: W' = bf16(W - lr * (grad o M)) o M, with the sum exact in
    float64 (dyadic gradients with few bits), rounded to float32 and then to bf16 by torch;
    compressing W' with the same mask must give the updated buffer byte for byte."""
    import torch

    N, K = 200, 136
    W, mask, _ = _rand_case(N, K, 70, seed=11)
    g = np.random.default_rng(12)
    grad = (g.integers(-255, 256, size=(N, K)) * 2.0 ** -10).astype(np.float32)
    lr = 2.0 ** -3
    buf, off = oracle.compress(W, mask)
    out = oracle.masked_update_bf16(buf, off, N, K, grad, lr)
    w64 = synth.bf16_to_f32(W).astype(np.float64)
    new32 = (w64 - lr * grad.astype(np.float64)).astype(np.float32)
    new_bits = torch.from_numpy(new32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    expect_buf, expect_off = oracle.compress(np.where(mask != 0, new_bits, 0).astype(np.uint16), mask)
    assert np.array_equal(expect_off, off)
    assert np.array_equal(out, expect_buf)


def test_masked_update_ignores_masked_out_gradient_and_zero_step(oracle):
    N, K = 130, 72
    W, mask, _ = _rand_case(N, K, 60, seed=13)
    g = np.random.default_rng(14).standard_normal((N, K)).astype(np.float32)
    buf, off = oracle.compress(W, mask)
    noisy = np.where(mask != 0, g, np.float32(3e38)).astype(np.float32)
    clean = np.where(mask != 0, g, np.float32(0)).astype(np.float32)
    a = oracle.masked_update_bf16(buf, off, N, K, noisy, 0.01)
    assert np.array_equal(a, oracle.masked_update_bf16(buf, off, N, K, clean, 0.01))
    assert not np.array_equal(a, buf)
    assert np.array_equal(oracle.masked_update_bf16(buf, off, N, K, noisy, 0.0), buf)


# ---------------------------------------------------------------- input generator


@pytest.mark.parametrize("K", [4096, 11008])
@pytest.mark.parametrize("pct,expect_nnz", [(50, None), (60, None), (70, None), (80, None)])
def test_mask_counts_exact(K, pct, expect_nnz):
    table = {4096: {50: 2048, 60: 1638, 70: 1229, 80: 819}, 11008: {50: 5504, 60: 4403, 70: 3302, 80: 2202}}
    g = np.random.default_rng(K + pct)
    W = synth.weight(8, K, g)
    mask = synth.magnitude_mask(W, pct)
    assert (mask.sum(axis=1) == table[K][pct]).all()
    # the kept entries are the largest |w| of each row
    a = np.abs(synth.bf16_to_f32(W))
    for r in range(8):
        assert a[r][mask[r] == 1].min() >= a[r][mask[r] == 0].max()


def test_nonuniform_mask_counts_and_outliers():
    K = 4096
    g = np.random.default_rng(0)
    W = synth.weight(64, K, g)
    mask, n_prune, outl = synth.nonuniform_mask(W, 70, np.random.default_rng(1))
    assert outl.size == 205 and np.unique(outl).size == 205
    assert (mask[:, outl] == 1).all()
    assert np.array_equal(mask.sum(axis=1), K - n_prune)
    assert ((n_prune >= round(0.6 * K) - 1) & (n_prune <= round(0.8 * K) + 1)).all()


def test_bf16_rne_matches_torch():
    torch = pytest.importorskip("torch")
    g = np.random.default_rng(4)
    a = np.concatenate([g.standard_normal(10000).astype(np.float32) * 10,
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 65504.0, 1e-30, -3.4e38], np.float32)])
    ours = synth.bf16_from_f32(a)
    ref = torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_quantize_int8_properties():
    g = np.random.default_rng(8)
    W = synth.weight(50, 256, g)
    mask = synth.magnitude_mask(W, 70)
    mask[3] = 0
    q, s = synth.quantize_int8(W, mask)
    assert s[3] == 1.0 and not q[3].any()
    assert (np.abs(q).max(axis=1)[np.arange(50) != 3] == 127).all()
    assert not q[mask == 0].any()


def test_per_token_activation_quantization_recipe():
    """The harness's INT8 activations (symmetric absmax per token): the largest |x| of a row
    maps to +-127 exactly, every code is within [-127, 127], and dequantizing is within half
    a step of x; an all-zero row gets scale 1 and zero codes."""
    from paper_2405_03594_gb300 import synth

    x = synth.activations(6, 200, np.random.default_rng(0))
    x[5] = 0
    qx, sx = synth.quantize_activations_int8(x)
    xf = synth.bf16_to_f32(x).astype(np.float64)
    assert qx.dtype == np.int8 and sx.dtype == np.float32 and np.abs(qx.astype(int)).max() <= 127
    for m in range(5):
        j = np.abs(xf[m]).argmax()
        assert abs(int(qx[m, j])) == 127
        assert np.abs(qx[m] * np.float64(sx[m]) - xf[m]).max() <= 0.5 * sx[m] * (1 + 1e-6)
    assert sx[5] == 1 and not qx[5].any()



def test_layer_sparsity_profile():
    """The per-layer profile: five levels within +-10 points of 70 %, mean exactly 70 %, as
    many layers as asked, the same for the same seed."""
    from paper_2405_03594_gb300 import synth

    for n in (4, 8, 32, 40):
        p = synth.layer_sparsity_profile(n)
        assert len(p) == n and sum(p) == 70 * n and set(p) <= {60, 65, 70, 75, 80}
        assert p == synth.layer_sparsity_profile(n)
    assert set(synth.layer_sparsity_profile(32)) == {60, 65, 70, 75, 80}
