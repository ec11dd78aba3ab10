"""GPU INT8-weight, INT8-activation sparse linear (sp_linear_w8a8) against the W8A8 oracle.

The path widens x[m, k] = bf16_rne(qx[m, k] * sx[m]) and runs the INT8-weight linear on it,
so against the oracle's exact integer sum it carries one rounding per activation and one
per output: ~2.4e-3 relative Frobenius error, inside the 5e-3 bound."""
import ctypes

import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2405_03594_gb300 import sp as _sp

    return _sp


def _int8_matrix(sp, N, K, pct, seed):
    W = synth.weight(N, K, np.random.default_rng(seed))
    mask = synth.magnitude_mask(W, pct)
    q, s = synth.quantize_int8(W, mask)
    return q, s, mask, sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(s))


def _acts(M, K, seed):
    return synth.quantize_activations_int8(synth.activations(M, K, np.random.default_rng(seed)))


def _run(h, qx, sx):
    return gu.bf16_from_dev(h.linear_w8a8(gu.i8_to_dev(qx), gu.f32_to_dev(sx)))


@pytest.mark.parametrize("N,K", [(300, 200), (129, 4096), (1000, 1024)])
@pytest.mark.parametrize("M", [1, 3, 4, 5, 16, 17])
def test_w8a8_small_tolerance(sp, oracle, N, K, M):
    q, s, mask, h = _int8_matrix(sp, N, K, 70, N + K)
    qx, sx = _acts(M, K, M)
    _, ref = oracle.linear_w8a8(qx, sx, q, mask, s)
    gu.assert_close(_run(h, qx, sx), ref, f"w8a8 {N}x{K} M={M}")
    sp.check()


@pytest.mark.parametrize("M", [2, 12, 40])
def test_w8a8_integer_inputs_bit_exact(sp, oracle, M):
    """Unit scales and small integers: the widened x is exact, every partial sum is an
    integer below 2^24, so y must be the bf16 rounding of the oracle's exact int64 sum."""
    N, K = 257, 1024
    g = np.random.default_rng(7)
    q = g.integers(-4, 5, size=(N, K)).astype(np.int8)
    mask = (g.random((N, K)) < 0.3).astype(np.uint8)
    q[mask == 0] = 0
    s = np.ones(N, dtype=np.float32)
    h = sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(s))
    qx = g.integers(-4, 5, size=(M, K)).astype(np.int8)
    sx = np.ones(M, dtype=np.float32)
    acc, _ = oracle.linear_w8a8(qx, sx, q, mask, s)
    y = gu.bf16_bits_from_dev(h.linear_w8a8(gu.i8_to_dev(qx), gu.f32_to_dev(sx)))
    assert np.array_equal(y, synth.bf16_from_f32(acc.astype(np.float32)))
    sp.check()


def test_w8a8_equals_int8_linear_on_widened_x(sp):
    """The call is the widening followed by the INT8-weight linear: widening on the host
    (float32 product, round to nearest even) and calling sp_linear gives the same bits."""
    q, s, mask, h = _int8_matrix(sp, 1000, 1024, 60, 3)
    for M in (1, 4, 9, 32):
        qx, sx = _acts(M, 1024, 10 + M)
        xw = synth.bf16_from_f32(qx.astype(np.float32) * sx[:, None])
        y1 = gu.bf16_bits_from_dev(h.linear_w8a8(gu.i8_to_dev(qx), gu.f32_to_dev(sx)))
        y2 = gu.bf16_bits_from_dev(h.linear(gu.bf16_to_dev(xw)))
        assert np.array_equal(y1, y2), M
    sp.check()


@pytest.mark.parametrize("name", list(synth.LLAMA2_7B_SHAPES))
def test_w8a8_llama_shapes_70pct(sp, oracle, name):
    N, K = synth.LLAMA2_7B_SHAPES[name]
    p = synth.PROJ_IDS[name]
    W = synth.weight(N, K, synth.rng(0, 0, p, synth.STREAM_W))
    mask = synth.magnitude_mask(W, 70)
    q, s = synth.quantize_int8(W, mask)
    h = sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(s))
    for M in (1, 16):
        qx, sx = synth.quantize_activations_int8(synth.activations(M, K, synth.rng(0, 0, p, synth.STREAM_X)))
        _, ref = oracle.linear_w8a8(qx, sx, q, mask, s)
        gu.assert_close(_run(h, qx, sx), ref, f"w8a8 {name} M={M}")
    sp.check()


def test_w8a8_workspace_shared_with_sp_linear(sp):
    """One zero-filled buffer serves sp_linear and sp_linear_w8a8 calls of different batch
    sizes in turn (the widened activations never land on sp_linear's counters)."""
    import torch

    q, s, mask, h = _int8_matrix(sp, 1000, 1024, 70, 5)
    big = max(h.w8a8_workspace_size(64), h.workspace_size(64))
    ws = torch.zeros(big, dtype=torch.uint8, device=gu.dev())
    for M in (64, 1, 16, 3):
        qx, sx = _acts(M, 1024, 20 + M)
        qd, sd = gu.i8_to_dev(qx), gu.f32_to_dev(sx)
        xw = gu.bf16_to_dev(synth.bf16_from_f32(qx.astype(np.float32) * sx[:, None]))
        w_shared = gu.bf16_bits_from_dev(h.linear_w8a8(qd, sd, workspace=ws))
        l_shared = gu.bf16_bits_from_dev(h.linear(xw, workspace=ws))
        w_fresh = gu.bf16_bits_from_dev(
            h.linear_w8a8(qd, sd, workspace=torch.zeros(big, dtype=torch.uint8, device=gu.dev())))
        l_fresh = gu.bf16_bits_from_dev(h.linear(xw, workspace=torch.zeros(big, dtype=torch.uint8, device=gu.dev())))
        assert np.array_equal(w_shared, w_fresh) and np.array_equal(l_shared, l_fresh), M
        assert np.array_equal(w_fresh, l_fresh), M
    sp.check()


def test_w8a8_argument_errors(sp):
    import torch

    lib = sp._lib
    q, s, mask, h = _int8_matrix(sp, 130, 72, 50, 1)
    qx, sx = _acts(4, 72, 1)
    qd, sd = gu.i8_to_dev(qx), gu.f32_to_dev(sx)
    y = torch.empty((4, 130), dtype=torch.bfloat16, device=gu.dev())
    need = h.w8a8_workspace_size(4)
    assert need >= h.workspace_size(4) + 4 * 72 * 2
    ws = torch.zeros(need, dtype=torch.uint8, device=gu.dev())
    P = ctypes.c_void_p
    call = lambda hh, qp, m, wsb: lib.sp_linear_w8a8(hh, P(qp), P(sd.data_ptr()), m, P(y.data_ptr()),
                                                     P(ws.data_ptr()), wsb, None)
    assert call(h.handle, qd.data_ptr(), 0, need) == 0  # m == 0: nothing to do
    assert call(h.handle, qd.data_ptr(), 4, need - 1) == 8  # workspace too small
    assert call(h.handle, qd.data_ptr() + 8, 4, need) == 3  # misaligned activations
    assert call(None, qd.data_ptr(), 4, need) == 7
    W = synth.weight(130, 72, np.random.default_rng(2))
    hb = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    assert call(hb.handle, qd.data_ptr(), 4, need) == 2  # bf16 handle: unsupported
    torch.cuda.synchronize()
