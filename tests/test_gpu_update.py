"""GPU masked weight update (Algorithm 1's step on the compressed form) against the oracle.

Both sides compute w <- bf16_rne(fma(-lr, g, w)) in float32 on every kept weight, so the
updated buffers must agree byte for byte (masks, offsets and padding included)."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2405_03594_gb300 import sp as _sp

    return _sp


def _case(N, K, pct, seed):
    g = np.random.default_rng(seed)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    grad = g.standard_normal((N, K), dtype=np.float32)
    return W, mask, grad


def _update_both(sp, oracle, W, mask, grad, lrs):
    N, K = W.shape
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    buf, off = oracle.compress(W, mask)
    gd = gu.f32_to_dev(grad)
    for lr in lrs:
        h.masked_update(gd, lr)
        buf = oracle.masked_update_bf16(buf, off, N, K, grad, lr)
    sp.check()
    got, goff = h.copy_out()
    return h, got, goff, buf, off


@pytest.mark.parametrize("N,K", [(1, 8), (130, 72), (300, 200), (257, 136), (129, 4096)])
@pytest.mark.parametrize("pct", [0, 50, 70, 95, 100])
def test_update_bytes_equal_oracle(sp, oracle, N, K, pct):
    W, mask, grad = _case(N, K, pct, N * 7 + K + pct)
    _, got, goff, buf, off = _update_both(sp, oracle, W, mask, grad, [0.01])
    assert np.array_equal(goff, off)
    assert np.array_equal(got, buf)


def test_two_steps_and_large_step(sp, oracle):
    W, mask, grad = _case(513, 1000, 60, 11)
    _, got, _, buf, _ = _update_both(sp, oracle, W, mask, grad, [0.5, 0.003])
    assert np.array_equal(got, buf)


def test_ties_to_even_on_gpu(sp, oracle):
    """Exact halfway results: w = 1 + m*2^-7 plus 2^-8 lies halfway between two bf16 values
    and must round to the one with an even last bit (both parities of m appear)."""
    N, K = 128, 64
    W = np.zeros((N, K), dtype=np.uint16)
    m = np.arange(N * K, dtype=np.int64).reshape(N, K) % 64
    W[:] = (0x3F80 + m).astype(np.uint16)  # 1 + m * 2^-7, exact in bf16
    mask = np.ones((N, K), dtype=np.uint8)
    grad = np.full((N, K), -1.0, dtype=np.float32)  # -lr * g = +2^-8 with lr = 2^-8
    _, got, _, buf, off = _update_both(sp, oracle, W, mask, grad, [2.0 ** -8])
    assert np.array_equal(got, buf)
    vals = np.frombuffer(buf[1024:1024 + 2 * N * K].tobytes(), dtype="<u2").reshape(N, K)
    expect = (0x3F80 + m + (m & 1)).astype(np.uint16)  # odd m rounds up, even m stays
    assert np.array_equal(vals, expect)


def test_masked_out_gradient_is_never_read(sp, oracle):
    """NaN in every masked-out gradient entry changes nothing: the step only touches kept
    weights (Algorithm 1 multiplies the gradient by the mask)."""
    W, mask, grad = _case(300, 200, 70, 5)
    poisoned = np.where(mask != 0, grad, np.float32(np.nan)).astype(np.float32)
    _, got, _, buf, _ = _update_both(sp, oracle, W, mask, poisoned, [0.02])
    _, _, _, clean, _ = _update_both(sp, oracle, W, mask, grad, [0.02])
    assert np.array_equal(got, clean)
    assert np.array_equal(buf, clean)


def test_zero_step_changes_nothing(sp, oracle):
    W, mask, grad = _case(257, 136, 50, 3)
    h, got, _, _, _ = _update_both(sp, oracle, W, mask, grad, [0.0])
    obuf, _ = oracle.compress(W, mask)
    assert np.array_equal(got, obuf)


def test_updated_handle_runs_linear(sp, oracle):
    """After a step the handle is an ordinary compressed matrix: decompress gives the
    updated masked weight and sp_linear matches the oracle product with it."""
    import torch

    N, K, M = 1000, 1024, 4
    W, mask, grad = _case(N, K, 70, 9)
    h, got, goff, buf, off = _update_both(sp, oracle, W, mask, grad, [0.01])
    Wn = oracle.decompress(buf, off, N, K, np.uint16)
    dense = gu.bf16_bits_from_dev(h.decompress())
    torch.cuda.synchronize()
    assert np.array_equal(dense, Wn)
    x = synth.activations(M, K, np.random.default_rng(2))
    y = h.linear(gu.bf16_to_dev(x))
    gu.assert_close(gu.bf16_from_dev(y), oracle.linear_bf16(x, Wn, mask), "linear after update")


@pytest.mark.parametrize("M,path", [(1, "cuda_core"), (4, "cuda_core"), (32, "tensor_core")])
def test_update_then_linear_on_one_stream_without_host_sync(sp, oracle, M, path):
    """Steps and products queued back to back on one stream, the host never waiting in
    between: each product must see the weights of the step just before it.  (The decode
    kernels copy their first weight chunks before waiting on the previous grid, so the
    launch right after an in-place update has to wait for it in full.)  A large step size
    makes a stale read show in the outputs."""
    import torch

    N, K = 4096, 4096
    W, mask, grad = _case(N, K, 70, 31)
    x = synth.activations(M, K, np.random.default_rng(5))
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    xd, gd = gu.bf16_to_dev(x), gu.f32_to_dev(grad)
    ws = torch.zeros(max(h.workspace_size(M), 256), dtype=torch.uint8, device=gu.dev())
    torch.cuda.synchronize()
    ys = []
    for _ in range(3):
        h.masked_update(gd, 0.5)
        y = torch.empty((M, N), dtype=torch.bfloat16, device=gu.dev())
        h.linear(xd, out=y, workspace=ws, path=path)
        ys.append(y)
    sp.check()
    buf, off = oracle.compress(W, mask)
    for i, y in enumerate(ys):
        buf = oracle.masked_update_bf16(buf, off, N, K, grad, 0.5)
        Wi = oracle.decompress(buf, off, N, K, np.uint16)
        gu.assert_close(gu.bf16_from_dev(y), oracle.linear_bf16(x, Wi, mask), f"product after step {i + 1}")


def test_gate_up_shape_70pct(sp, oracle):
    """The largest Llama-2-7B shape (gate/up 22016 x 4096) at 70 %: every updated byte."""
    name = "gate_up"
    N, K = synth.LLAMA2_7B_SHAPES[name]
    W = synth.weight(N, K, synth.rng(0, 0, 2, synth.STREAM_W))
    mask = synth.magnitude_mask(W, 70)
    grad = np.random.default_rng(4).standard_normal((N, K), dtype=np.float32)
    _, got, _, buf, _ = _update_both(sp, oracle, W, mask, grad, [1e-3])
    assert np.array_equal(got, buf)


def test_argument_errors(sp):
    import torch

    W, mask, grad = _case(130, 72, 50, 1)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    gd = gu.f32_to_dev(grad)
    lib = sp._lib
    import ctypes

    assert lib.sp_masked_update(h.handle, None, ctypes.c_float(0.1), None) == 1  # null gradient
    assert lib.sp_masked_update(h.handle, ctypes.c_void_p(gd.data_ptr()), ctypes.c_float(float("nan")), None) == 1
    assert lib.sp_masked_update(h.handle, ctypes.c_void_p(gd.data_ptr()), ctypes.c_float(float("inf")), None) == 1
    assert lib.sp_masked_update(h.handle, ctypes.c_void_p(gd.data_ptr() + 4), ctypes.c_float(0.1), None) == 3
    q, s = synth.quantize_int8(W, mask)
    hi = sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(s))
    assert lib.sp_masked_update(hi.handle, ctypes.c_void_p(gd.data_ptr()), ctypes.c_float(0.1), None) == 2
    torch.cuda.synchronize()
