"""GPU sparse linear through the C ABI against the float64 oracle.

Tolerances (acceptance bar): max|err| <= 1e-2 * max|ref|, relative Frobenius <= 5e-3.
Bit-exact where the arithmetic is exact: integer-valued inputs, one-hot x, empty rows."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

PATHS = ["cuda_core", "tensor_core"]


@pytest.fixture(scope="module")
def sp():
    from paper_2405_03594_gb300 import sp as _sp

    return _sp


def _case(N, K, M, pct, seed, int8=False):
    g = np.random.default_rng(seed)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    x = synth.activations(M, K, g)
    if int8:
        q, s = synth.quantize_int8(W, mask)
        return q, s, mask, x
    return W, None, mask, x


def _run(sp, vals, s, mask, x, path="auto"):
    if s is not None:
        h = sp.compress(gu.i8_to_dev(vals), gu.u8_to_dev(mask), gu.f32_to_dev(s))
    else:
        h = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
    y = h.linear(gu.bf16_to_dev(x), path=path)
    sp.check()
    return h, y


def _ref(oracle, vals, s, mask, x):
    if s is not None:
        return oracle.linear_int8(x, vals, mask, s)
    return oracle.linear_bf16(x, vals, mask)


SMALL = [(128, 64), (300, 200), (257, 136), (1000, 1024), (130, 4096), (64, 11008)]


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("N,K", SMALL)
@pytest.mark.parametrize("M", [1, 2, 3, 4, 5, 8, 9, 16])
@pytest.mark.parametrize("int8", [False, True])
def test_linear_small_tolerance(sp, oracle, path, N, K, M, int8):
    vals, s, mask, x = _case(N, K, M, 70, seed=N + K + M, int8=int8)
    _, y = _run(sp, vals, s, mask, x, path)
    gu.assert_close(gu.bf16_from_dev(y), _ref(oracle, vals, s, mask, x), f"{N}x{K} M={M}")


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("pct", [0, 50, 60, 80, 95])
def test_linear_sparsity_levels(sp, oracle, path, pct):
    vals, s, mask, x = _case(700, 520, 4, pct, seed=pct)
    _, y = _run(sp, vals, s, mask, x, path)
    gu.assert_close(gu.bf16_from_dev(y), _ref(oracle, vals, s, mask, x), f"{pct}%")


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("N,K,M", [(300, 200, 3), (1000, 1024, 8), (129, 4096, 16), (256, 11008, 1)])
@pytest.mark.parametrize("int8", [False, True])
def test_integer_inputs_bit_exact(sp, oracle, path, N, K, M, int8):
    """x in {-2..2}, W in {-4..4} (INT8: q in {-127..127}, s = 1): every FP32 partial sum is
    an integer below 2^24, so the GPU result must be the bf16 rounding of the exact sum."""
    g = np.random.default_rng(N * K + M)
    mask = (g.random((N, K)) < 0.35).astype(np.uint8)
    x = synth.bf16_from_f32(g.integers(-2, 3, size=(M, K)).astype(np.float32))
    if int8:
        q = (g.integers(-127, 128, size=(N, K)) * mask).astype(np.int8)
        s = np.ones(N, dtype=np.float32)
        _, y = _run(sp, q, s, mask, x, path)
        ref = oracle.linear_int8(x, q, mask, s)
        assert np.abs(ref).max() < 2**24
    else:
        W = synth.bf16_from_f32(g.integers(-4, 5, size=(N, K)).astype(np.float32))
        _, y = _run(sp, W, None, mask, x, path)
        ref = oracle.linear_bf16(x, W, mask)
    expect = synth.bf16_from_f32(ref.astype(np.float32))
    assert np.array_equal(gu.bf16_bits_from_dev(y), expect)


@pytest.mark.parametrize("path", PATHS)
def test_one_hot_rows_select_columns_bit_exact(sp, oracle, path):
    N, K = 300, 200
    vals, _, mask, _ = _case(N, K, 1, 50, seed=3)
    ks = [0, 1, 31, 32, 33, 63, 64, 127, 128, 191, 192, 199]
    x = np.zeros((len(ks), K), dtype=np.uint16)
    for i, k in enumerate(ks):
        x[i, k] = 0x3F80
    h = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
    for m0 in range(0, len(ks), 4):
        y = h.linear(gu.bf16_to_dev(x[m0:m0 + 4]), path=path)
        got = gu.bf16_bits_from_dev(y)
        for i, k in enumerate(ks[m0:m0 + 4]):
            assert np.array_equal(got[i], np.where(mask[:, k] != 0, vals[:, k], 0).astype(np.uint16)), k
    sp.check()


@pytest.mark.parametrize("path", PATHS)
def test_empty_rows_and_all_pruned(sp, oracle, path):
    vals, _, mask, x = _case(260, 136, 3, 50, seed=4)
    mask[[0, 127, 128, 259]] = 0
    _, y = _run(sp, vals, None, mask, x, path)
    got = gu.bf16_bits_from_dev(y)
    assert not got[:, [0, 127, 128, 259]].any()
    empty = np.zeros_like(mask)
    _, y0 = _run(sp, vals, None, empty, x, path)
    assert not gu.bf16_bits_from_dev(y0).any()


@pytest.mark.parametrize("path", PATHS)
def test_dense_reduces_to_library_matmul(sp, oracle, path):
    """0% sparsity is a plain dense matmul: compare with torch's float64 CPU matmul."""
    import torch

    vals, _, mask, x = _case(384, 320, 5, 0, seed=6)
    assert mask.all()
    _, y = _run(sp, vals, None, mask, x, path)
    ref = (torch.from_numpy(synth.bf16_to_f32(x).astype(np.float64)) @
           torch.from_numpy(synth.bf16_to_f32(vals).astype(np.float64)).T).numpy()
    gu.assert_close(gu.bf16_from_dev(y), ref, "dense")


@pytest.mark.parametrize("path", PATHS)
def test_bitwise_repeatable(sp, oracle, path):
    vals, _, mask, x = _case(4096, 4096, 4, 70, seed=7)
    h = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
    xd = gu.bf16_to_dev(x)
    a = gu.bf16_bits_from_dev(h.linear(xd, path=path))
    for _ in range(3):
        b = gu.bf16_bits_from_dev(h.linear(xd, path=path))
        assert np.array_equal(a, b)


def test_m_zero_is_a_no_op(sp):
    import torch

    vals, _, mask, _ = _case(128, 64, 1, 50, seed=8)
    h = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
    x = torch.empty((0, 64), dtype=torch.bfloat16, device="cuda")
    y = h.linear(x)
    assert y.shape == (0, 128)
    sp.check()


def test_workspace_too_small_is_rejected(sp):
    import torch

    vals, _, mask, x = _case(300, 200, 2, 50, seed=9)
    h = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
    ws = torch.zeros(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(sp.SpError) as e:
        h.linear(gu.bf16_to_dev(x), workspace=ws)
    assert e.value.code == 8


# ------------------------------------------------------------------ full-size configurations


def test_config_q_proj_4096_50pct_m16_seed0(sp, oracle):
    """Single 4096x4096 layer, 50% per-row magnitude sparsity, x [16, 4096], seed 0."""
    W, mask, x = synth.layer_inputs("o", 50, 16, seed=0)
    assert (mask.sum(axis=1) == 2048).all()
    _, y = _run(sp, W, None, mask, x)
    gu.assert_close(gu.bf16_from_dev(y), oracle.linear_bf16(x, W, mask), "q_proj 50% M=16")


@pytest.mark.parametrize("name", list(synth.LLAMA2_7B_SHAPES))
def test_config_llama_shapes_70pct_decode(sp, oracle, name):
    W, mask, x16 = synth.layer_inputs(name, 70, 16, seed=0)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    ref16 = oracle.linear_bf16(x16, W, mask)
    for M in (1, 4, 16):
        y = h.linear(gu.bf16_to_dev(x16[:M]))
        gu.assert_close(gu.bf16_from_dev(y), ref16[:M], f"{name} M={M}")
    sp.check()


@pytest.mark.parametrize("name", list(synth.LLAMA2_7B_SHAPES))
@pytest.mark.parametrize("pct", [50, 70])
def test_config_prefill_2048_sampled(sp, oracle, name, pct):
    """Prefill: the four shapes at 50% and 70%, x [2048, K], on the tensor-core kernel with
    the inputs and launch the bench's prefill section times; the oracle computes 64 output
    rows (all 2048 tokens each), the first and last included."""
    W, mask, _ = synth.layer_inputs(name, pct, 1, seed=0, layer=0)
    N, K = W.shape
    x = synth.activations(2048, K, synth.rng(0, 0, synth.PROJ_IDS[name], synth.STREAM_X))
    _, y = _run(sp, W, None, mask, x, path="tensor_core")
    rows = np.sort(np.random.default_rng(pct + N).choice(N, 64, replace=False))
    rows[0], rows[-1] = 0, N - 1
    ref = oracle.linear_bf16(x, W[rows], mask[rows])
    import torch

    got = gu.bf16_from_dev(y[:, torch.from_numpy(rows).to(y.device)])
    gu.assert_close(got, ref, f"prefill {name} {pct}% M=2048")
    # every output row for eight tokens (first, last, six random): every row block, every
    # stream-K fix-up and every TMA-store tile of the launch
    toks = np.sort(np.random.default_rng(pct * 7 + N).choice(np.arange(1, 2047), 6, replace=False))
    toks = np.concatenate([[0], toks, [2047]])
    ref_t = oracle.linear_bf16(np.ascontiguousarray(x[toks]), W, mask)
    got_t = gu.bf16_from_dev(y[torch.from_numpy(toks).to(y.device)])
    gu.assert_close(got_t, ref_t, f"prefill {name} {pct}% M=2048, all rows of tokens {toks.tolist()}")


@pytest.mark.parametrize("name", ["gate_up", "down"])
@pytest.mark.parametrize("pct", [0, 50, 60, 70, 80])
def test_config_sweep_nonuniform_sampled(sp, oracle, name, pct):
    """Non-uniform masks (per-row sparsity within +-10 points, 5% dense columns), M up to
    256; the oracle computes a sample of 192 output rows."""
    N, K = synth.LLAMA2_7B_SHAPES[name]
    p = synth.PROJ_IDS[name]
    W = synth.weight(N, K, synth.rng(0, 0, p, synth.STREAM_W))
    mask, n_prune, _ = synth.nonuniform_mask(W, pct, synth.rng(0, 0, p, synth.STREAM_MASK))
    assert np.array_equal(mask.sum(axis=1), K - n_prune)
    x = synth.activations(256, K, synth.rng(0, 0, p, synth.STREAM_X))
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    rows = np.sort(np.random.default_rng(pct).choice(N, 192, replace=False))
    rows[0], rows[-1] = 0, N - 1
    ref = oracle.linear_bf16(x, W[rows], mask[rows])
    # every output row for a few tokens of each batch size (all tokens up to M = 8; else the
    # first, the last and six random ones); the oracle runs once on the union of those tokens
    rng = np.random.default_rng(pct + 11)
    toks_by_m = {}
    for M in (1, 2, 4, 8, 16, 32, 64, 128, 256):
        toks_by_m[M] = (np.arange(M) if M <= 8 else
                        np.concatenate([[0], np.sort(rng.choice(np.arange(1, M - 1), 6, replace=False)), [M - 1]]))
    union = np.unique(np.concatenate(list(toks_by_m.values())))
    ref_u = oracle.linear_bf16(np.ascontiguousarray(x[union]), W, mask)
    pos = {int(tk): i for i, tk in enumerate(union)}
    for M in (1, 2, 4, 8, 16, 32, 64, 128, 256):
        y = gu.bf16_from_dev(h.linear(gu.bf16_to_dev(x[:M])))
        gu.assert_close(y[:, rows], ref[:M], f"{name} {pct}% M={M}")
        tk = toks_by_m[M]
        gu.assert_close(y[tk], ref_u[[pos[int(v)] for v in tk]], f"{name} {pct}% M={M}, all rows of tokens {tk.tolist()}")
    sp.check()


@pytest.mark.parametrize("N,K", [(4096, 64), (2000, 128), (1500, 200), (700, 1024)])
@pytest.mark.parametrize("M", [17, 100, 256, 300])
def test_tensor_core_short_segments(sp, oracle, N, K, M):
    """Tensor-core path with few K-tiles per row block (T = 1 .. 16): every CTA's range
    covers many short (token tile, row block) segments, so an expander warpgroup can
    finish a segment before the MMA issuer has finished the previous one on the same
    accumulator; wide token tiles (up to 256 tokens) and a ragged last token tile."""
    vals, s, mask, x = _case(N, K, M, 70, seed=N + K + M)
    _, y = _run(sp, vals, s, mask, x, "tensor_core")
    gu.assert_close(gu.bf16_from_dev(y), _ref(oracle, vals, s, mask, x), f"{N}x{K} M={M}")


def test_launch_count(sp):
    """sp_launch_count: one launch per 16 rows on the CUDA-core family, one on the tensor-core
    family, and AUTO switches at M = 11 for bf16 values and at M = 14 for int8 values."""
    vals, s, mask, _ = _case(300, 200, 1, 70, seed=5)
    h = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
    q, sc = __import__("paper_2405_03594_gb300").synth.quantize_int8(vals, mask)
    h8 = sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(sc))
    assert h.launch_count(0) == 0
    assert [h.launch_count(m, "cuda_core") for m in (1, 16, 17, 40)] == [1, 1, 2, 3]
    assert [h.launch_count(m, "tensor_core") for m in (1, 16, 17, 300)] == [1, 1, 1, 1]
    assert [h.launch_count(m) for m in (1, 10, 11, 40)] == [1, 1, 1, 1]
    assert [h8.launch_count(m) for m in (13, 14, 17)] == [1, 1, 1]
    assert h8.launch_count(40, "cuda_core") == 3
    with pytest.raises(sp.SpError):
        h.launch_count(-1)
    assert h.kernel_name(1) == "linear_ccw_kernel" and h.kernel_name(8) == "linear_cc_kernel"
    assert h.kernel_name(11) == "linear_tc_kernel" and h.kernel_name(3, "tensor_core") == "linear_tc_kernel"


def test_shared_workspace_across_grids(sp, oracle):
    """Matrices whose launches use different grid sizes share one workspace, interleaved:
    the split-K counters must never be overlaid by another call's partials."""
    import torch

    cases = [_case(N, K, M, 70, seed=N + M) for N, K, M in
             [(257, 136, 2), (64, 11008, 1), (1000, 1024, 2), (4096, 4096, 3), (130, 4096, 5)]]
    hs = [sp.compress(gu.bf16_to_dev(v), gu.u8_to_dev(m)) for v, _, m, _ in cases]
    need = max(h.workspace_size(c[3].shape[0]) for h, c in zip(hs, cases))
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    refs = [oracle.linear_bf16(x, v, m) for v, _, m, x in cases]
    for rep in range(3):
        for h, (v, _, m, x), ref in zip(hs, cases, refs):
            y = gu.bf16_from_dev(h.linear(gu.bf16_to_dev(x), workspace=ws))
            gu.assert_close(y, ref, f"rep {rep} N={v.shape[0]}")
    sp.check()


@pytest.mark.parametrize("pct", [50, 90])
def test_square_12288_prefill_parity(sp, oracle, pct):
    """The 12K x 12K sparse matmul of the sparsity-scaling example (Sec. 2.3), at M = 2048 on
    the tensor-core kernel as the bench's square sweep runs it: 64 sampled output rows over
    all tokens (first and last rows included), and every output row for 8 tokens."""
    import torch

    N = K = 12288
    W = synth.weight(N, K, synth.rng(0, 0, 0, synth.STREAM_W))
    mask = synth.magnitude_mask(W, pct)
    x = synth.activations(2048, K, synth.rng(0, 0, 0, synth.STREAM_X))
    _, y = _run(sp, W, None, mask, x, path="tensor_core")
    rows = np.sort(np.random.default_rng(pct).choice(N, 64, replace=False))
    rows[0], rows[-1] = 0, N - 1
    ref = oracle.linear_bf16(x, W[rows], mask[rows])
    got = gu.bf16_from_dev(y[:, torch.from_numpy(rows).to(y.device)])
    gu.assert_close(got, ref, f"12288^2 {pct}% M=2048, sampled rows")
    toks = np.concatenate([[0], np.sort(np.random.default_rng(pct + 1).choice(np.arange(1, 2047), 6, replace=False)),
                           [2047]])
    ref_t = oracle.linear_bf16(np.ascontiguousarray(x[toks]), W, mask)
    gu.assert_close(gu.bf16_from_dev(y[torch.from_numpy(toks).to(y.device)]), ref_t,
                    f"12288^2 {pct}% M=2048, all rows of tokens {toks.tolist()}")
